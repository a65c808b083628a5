// relation_layer.cu -- the layer's transforms around the operator (Sec. 3.1-3.2,
// Eq. givens-rotation, App. A.2.2, App. B.3), as a producer pass in front of the
// Relation kernels and its gradient pass behind them.
//
//   RoPE (full head, RoFormer's interleaved pairs): pair c of the row at position m
//   (zero-based within its sequence) turns by m * base^(-2c/d):
//       (x_2c, x_2c+1) -> (x_2c cos - x_2c+1 sin, x_2c sin + x_2c+1 cos)
//   applied to P1 -> Q and P2 -> K; the information states are not rotated.
//   Givens mixing of head pairs (a, b) with angle theta_k, on every channel:
//       I~_a = cos I_a - sin I_b,   I~_b = sin I_a + cos I_b   (V = I~)
//   pairing A: (0,1), (2,3), ...; pairing B: (1,2), (3,4), ..., (H-1,0).
//   Gradients: the transposed rotations, and
//       dtheta_k = sum dI~_a (-sin I_a - cos I_b) + dI~_b (cos I_a - sin I_b).
//
// Both passes are HBM-bound (prep reads P1, P2, I and writes Q, K, V; grad reads dQ, dK,
// dV, I and writes dP1, dP2, dI): one CTA per (sequence, 16 positions) moves 8-element
// vectors (16 bytes in bf16).  The rotation angles of the CTA's positions are tabulated
// once in shared memory and reused by every head: m * base^(-2c/d) is formed and reduced
// modulo 2 pi in fp64 (positions reach 16k, where an fp32 angle would be off by ~1e-3
// rad), then its cosine and sine are taken in fp32.  dtheta is summed per CTA in a fixed
// order and the partials are added up in fp64 by a second kernel, one block per head
// pair (deterministic).
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rel {
namespace layer {

constexpr int kTok = 16;       // positions per CTA
constexpr int kThreads = 256;
constexpr int kMaxD = 256;     // head size limit of these passes
constexpr int kMaxPairs = 128; // H / 2 limit

template <typename TI>
struct Vec8;
template <>
struct Vec8<__nv_bfloat16> {
  __device__ static void load(const void* p, float (&x)[8]) {
    const uint4 w = *reinterpret_cast<const uint4*>(p);
    const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u[i]));
      x[2 * i] = f.x;
      x[2 * i + 1] = f.y;
    }
  }
  __device__ static void store(void* p, const float (&x)[8]) {
    *reinterpret_cast<uint4*>(p) = make_uint4(pack_bf16x2(x[0], x[1]), pack_bf16x2(x[2], x[3]),
                                              pack_bf16x2(x[4], x[5]), pack_bf16x2(x[6], x[7]));
  }
};
template <>
struct Vec8<float> {
  __device__ static void load(const void* p, float (&x)[8]) {
    const float4 a = reinterpret_cast<const float4*>(p)[0];
    const float4 b = reinterpret_cast<const float4*>(p)[1];
    x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
    x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
  }
  __device__ static void store(void* p, const float (&x)[8]) {
    reinterpret_cast<float4*>(p)[0] = make_float4(x[0], x[1], x[2], x[3]);
    reinterpret_cast<float4*>(p)[1] = make_float4(x[4], x[5], x[6], x[7]);
  }
};

struct Tables {
  double w[kMaxD / 2];                             // base^(-2c/d), fp64
  float cs[kTok][kMaxD / 2], sn[kTok][kMaxD / 2];  // RoPE of the CTA's positions
  float tc[kMaxPairs], ts[kMaxPairs];              // cos, sin of the Givens angles
  float part[kThreads / 32][kMaxPairs];            // dtheta: per-warp partial sums
};

// cos / sin of m * base^(-2c/d) for the CTA's positions, and of the Givens angles.  The
// d/2 frequencies first (fp64 exp, the expensive part on this GPU's fp64 pipe), then
// per entry one fp64 product and a reduction modulo 2 pi.
__device__ void fill_tables(Tables& tb, const LayerProblem& p, int t0) {
  const int half = p.d / 2;
  const double lnb = log((double)p.rope_base);
  for (int c = threadIdx.x; c < half; c += kThreads)
    tb.w[c] = exp(-2.0 * (double)c / (double)p.d * lnb);
  __syncthreads();
  const double two_pi = 6.283185307179586476925286766559;
  const double inv_two_pi = 0.15915494309189533576888376337251;
  for (int e = threadIdx.x; e < kTok * half; e += kThreads) {
    const int tt = e / half, c = e % half;
    const double a = (double)(t0 + tt) * tb.w[c];
    const float r = (float)fma(-rint(a * inv_two_pi), two_pi, a);  // |r| <= pi (+ rounding)
    float s, co;
    sincosf(r, &s, &co);
    tb.cs[tt][c] = co;
    tb.sn[tt][c] = s;
  }
  for (int k = threadIdx.x; k < p.H / 2; k += kThreads) {
    float s, co;
    sincosf(p.theta[k], &s, &co);
    tb.tc[k] = co;
    tb.ts[k] = s;
  }
}

// heads of Givens pair k
__device__ __forceinline__ void pair_heads(const LayerProblem& p, int k, int& a, int& b) {
  a = p.pairing == 0 ? 2 * k : 2 * k + 1;
  b = p.pairing == 0 ? 2 * k + 1 : (2 * k + 2) % p.H;
}

// rotate the 4 pairs of an 8-element chunk starting at channel 8 u by +-angle
__device__ __forceinline__ void rotate8(float (&x)[8], const Tables& tb, int tt, int u,
                                        float sgn) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float co = tb.cs[tt][4 * u + i], s = sgn * tb.sn[tt][4 * u + i];
    const float x0 = x[2 * i], x1 = x[2 * i + 1];
    x[2 * i] = x0 * co - x1 * s;
    x[2 * i + 1] = x0 * s + x1 * co;
  }
}

// RoPE (sgn = +1) or its transpose (sgn = -1) of in1 -> out1 and in2 -> out2 over the
// CTA's (position, head, chunk) items, two items per thread and iteration so that four
// 16-byte loads are in flight.
template <typename TI>
__device__ __forceinline__ void rope_pass(const LayerProblem& p, const Tables& tb, int t0, int nt,
                                          float sgn) {
  const int nu = p.d / 8;
  const int n = nt * p.H * nu;
  const long long base = (long long)(blockIdx.x / ((p.T + kTok - 1) / kTok)) * p.sB;
  auto off_of = [&](int e, int& tt, int& u) {
    u = e % nu;
    const int h = (e / nu) % p.H;
    tt = e / (nu * p.H);
    return base + (long long)(t0 + tt) * p.sT + (long long)h * p.sH + 8 * u;
  };
  for (int e = threadIdx.x; e < n; e += 2 * kThreads) {
    const int e2 = e + kThreads;
    const bool two = e2 < n;
    int tt0, u0, tt1 = 0, u1 = 0;
    const long long o0 = off_of(e, tt0, u0);
    const long long o1 = two ? off_of(e2, tt1, u1) : o0;
    float x0[8], y0[8], x1[8], y1[8];
    Vec8<TI>::load(reinterpret_cast<const TI*>(p.in1) + o0, x0);
    Vec8<TI>::load(reinterpret_cast<const TI*>(p.in2) + o0, y0);
    Vec8<TI>::load(reinterpret_cast<const TI*>(p.in1) + o1, x1);
    Vec8<TI>::load(reinterpret_cast<const TI*>(p.in2) + o1, y1);
    rotate8(x0, tb, tt0, u0, sgn);
    rotate8(y0, tb, tt0, u0, sgn);
    Vec8<TI>::store(reinterpret_cast<TI*>(p.out1) + o0, x0);
    Vec8<TI>::store(reinterpret_cast<TI*>(p.out2) + o0, y0);
    if (two) {
      rotate8(x1, tb, tt1, u1, sgn);
      rotate8(y1, tb, tt1, u1, sgn);
      Vec8<TI>::store(reinterpret_cast<TI*>(p.out1) + o1, x1);
      Vec8<TI>::store(reinterpret_cast<TI*>(p.out2) + o1, y1);
    }
  }
}

template <typename TI>
__global__ void __launch_bounds__(kThreads) prep_kernel(LayerProblem p) {
  __shared__ Tables tb;
  const int n_tt = (p.T + kTok - 1) / kTok;
  const int b = blockIdx.x / n_tt, t0 = (blockIdx.x % n_tt) * kTok;
  const int nt = min(kTok, p.T - t0);
  fill_tables(tb, p, t0);
  __syncthreads();
  const int nu = p.d / 8;  // 8-element chunks per row
  const long long base = (long long)b * p.sB;
  rope_pass<TI>(p, tb, t0, nt, 1.f);  // Q = RoPE(P1), K = RoPE(P2)
  // Givens mixing of the information states: (token, pair, chunk) items
  const int np = p.H / 2;
  for (int e = threadIdx.x; e < nt * np * nu; e += kThreads) {
    const int u = e % nu, k = (e / nu) % np, tt = e / (nu * np);
    int ha, hb;
    pair_heads(p, k, ha, hb);
    const long long row = base + (long long)(t0 + tt) * p.sT + 8 * u;
    const long long oa = row + (long long)ha * p.sH, ob = row + (long long)hb * p.sH;
    float ia[8], ib[8], va[8], vb[8];
    Vec8<TI>::load(reinterpret_cast<const TI*>(p.in3) + oa, ia);
    Vec8<TI>::load(reinterpret_cast<const TI*>(p.in3) + ob, ib);
    const float co = tb.tc[k], s = tb.ts[k];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      va[i] = co * ia[i] - s * ib[i];
      vb[i] = s * ia[i] + co * ib[i];
    }
    Vec8<TI>::store(reinterpret_cast<TI*>(p.out3) + oa, va);
    Vec8<TI>::store(reinterpret_cast<TI*>(p.out3) + ob, vb);
  }
}

template <typename TI>
__global__ void __launch_bounds__(kThreads) grad_kernel(LayerProblem p) {
  __shared__ Tables tb;
  const int n_tt = (p.T + kTok - 1) / kTok;
  const int b = blockIdx.x / n_tt, t0 = (blockIdx.x % n_tt) * kTok;
  const int nt = min(kTok, p.T - t0);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  fill_tables(tb, p, t0);
  for (int k = lane; k < p.H / 2; k += 32) tb.part[warp][k] = 0.f;
  __syncthreads();
  const int nu = p.d / 8;
  const long long base = (long long)b * p.sB;
  rope_pass<TI>(p, tb, t0, nt, -1.f);  // transposed RoPE: dP1 from dQ, dP2 from dK
  // transposed Givens: dI from dV = dI~, and dtheta.  The loop runs the same number of
  // times on every lane (items past the end are idle), so the warp can reduce dtheta
  // over runs of lanes with the same pair (items are ordered chunk, pair, position) and
  // add each run's sum to its pair's slot in lane order (deterministic).
  const int np = p.H / 2;
  const int n_items = nt * np * nu;
  for (int e0 = 0; e0 < n_items; e0 += kThreads) {
    const int e = e0 + (int)threadIdx.x;
    const bool live = e < n_items;
    const int ec = live ? e : 0;
    const int u = ec % nu, k = (ec / nu) % np, tt = ec / (nu * np);
    float dt = 0.f;
    if (live) {
      int ha, hb;
      pair_heads(p, k, ha, hb);
      const long long row = base + (long long)(t0 + tt) * p.sT + 8 * u;
      const long long oa = row + (long long)ha * p.sH, ob = row + (long long)hb * p.sH;
      float ga[8], gb[8], ia[8], ib[8], da[8], db[8];
      Vec8<TI>::load(reinterpret_cast<const TI*>(p.in3) + oa, ga);
      Vec8<TI>::load(reinterpret_cast<const TI*>(p.in3) + ob, gb);
      Vec8<TI>::load(reinterpret_cast<const TI*>(p.in4) + oa, ia);
      Vec8<TI>::load(reinterpret_cast<const TI*>(p.in4) + ob, ib);
      const float co = tb.tc[k], s = tb.ts[k];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        da[i] = co * ga[i] + s * gb[i];
        db[i] = -s * ga[i] + co * gb[i];
        dt += ga[i] * (-s * ia[i] - co * ib[i]) + gb[i] * (co * ia[i] - s * ib[i]);
      }
      Vec8<TI>::store(reinterpret_cast<TI*>(p.out3) + oa, da);
      Vec8<TI>::store(reinterpret_cast<TI*>(p.out3) + ob, db);
    }
    // runs of consecutive lanes with the same pair (idle lanes form runs of their own)
    const int key = live ? k : -1 - lane;
    const int kprev = __shfl_up_sync(0xffffffffu, key, 1);
    const bool head = lane == 0 || kprev != key;
    const unsigned heads = __ballot_sync(0xffffffffu, head);
    const int first = 31 - __clz(heads & (0xffffffffu >> (31 - lane)));  // my run's first lane
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(0xffffffffu, dt, o);
      if (lane - o >= first) dt += t;
    }
    const int knext = __shfl_down_sync(0xffffffffu, key, 1);
    const bool tail = lane == 31 || knext != key;
    const int run = __popc(heads & (0xffffffffu >> (31 - lane))) - 1;
    const int n_runs = __popc(heads);
    for (int r = 0; r < n_runs; ++r) {
      if (tail && live && run == r) tb.part[warp][k] += dt;
      __syncwarp();
    }
  }
  __syncthreads();
  for (int k = threadIdx.x; k < np; k += kThreads) {
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) s += tb.part[w][k];
    p.dtheta_part[(long long)blockIdx.x * np + k] = s;
  }
}

// dtheta_k = sum over CTAs of the partials, in fp64 and a fixed order; one block per pair
__global__ void __launch_bounds__(256) dtheta_kernel(LayerProblem p, int n_cta) {
  __shared__ double red[256];
  const int np = p.H / 2, k = blockIdx.x;
  double s = 0.0;
  for (int c = threadIdx.x; c < n_cta; c += 256) s += (double)p.dtheta_part[(long long)c * np + k];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) p.dtheta[k] = (float)red[0];
}

int ctas(const LayerProblem& p) { return p.B * ((p.T + kTok - 1) / kTok); }

}  // namespace layer

bool layer_supports(relation_dtype dt, int d, int H) {
  return (dt == RELATION_F32 || dt == RELATION_BF16) && d >= 8 && d % 8 == 0 &&
         d <= layer::kMaxD && H >= 2 && H % 2 == 0 && H / 2 <= layer::kMaxPairs;
}

size_t layer_grad_workspace_bytes(int B, int T, int H) {
  return (size_t)B * ((T + layer::kTok - 1) / layer::kTok) * (H / 2) * sizeof(float);
}

cudaError_t launch_layer_prep(const LayerProblem& p, cudaStream_t s) {
  const int grid = layer::ctas(p);
  if (p.dtype == RELATION_F32)
    layer::prep_kernel<float><<<grid, layer::kThreads, 0, s>>>(p);
  else
    layer::prep_kernel<__nv_bfloat16><<<grid, layer::kThreads, 0, s>>>(p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) note_failure("layer prep: launch");
  return e;
}

cudaError_t launch_layer_grad(const LayerProblem& p, cudaStream_t s) {
  const int grid = layer::ctas(p);
  if (p.dtype == RELATION_F32)
    layer::grad_kernel<float><<<grid, layer::kThreads, 0, s>>>(p);
  else
    layer::grad_kernel<__nv_bfloat16><<<grid, layer::kThreads, 0, s>>>(p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { note_failure("layer grad: launch"); return e; }
  layer::dtheta_kernel<<<p.H / 2, 256, 0, s>>>(p, grid);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("layer grad: dtheta launch");
  return e;
}

}  // namespace rel
