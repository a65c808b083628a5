// relation_simt.cu -- CUDA-core (SIMT) FlashRelation kernels, fp32 and bf16 I/O.
//
// These kernels run the exact causal Relation operator with fp32 arithmetic on the
// CUDA cores.  They serve the fp32 workloads (accurate expf / logf / division, no
// approximate transcendental instructions) and every (dtype, d_h) the tensor-core
// kernels do not cover.
//
// Forward (Sec. 5.1, App. A.3): one CTA owns 64 query rows of one head; 4 threads
// share a row, each holding a quarter of q_i and of the Exchange accumulator z.  Key
// and value tiles of 64 rows are staged in shared memory as fp32.  Per tile the row's
// Exchange entries E_ij = SiLU(U_ij) (j < i) update the running (m, l, z) state; the
// diagonal entry gives S_i = sigmoid(U_ii / tau_S) and is kept out of the scan.  The
// epilogue applies the count correction and the Self-Exchange split:
//   A_i = m + log l - lambda log i, g_i = sigmoid(A_i - S_i),
//   Y_i = (1 - g_i) v_i + g_i z / l,  logZ_i = logaddexp(S_i, A_i)   (App. A.3.5).
//
// Backward (App. A.1.7): the Self part and D_i come from the shared row kernel
// (bwd_common.cu); a key-stationary kernel accumulates dK, dV over query tiles and a
// query-stationary kernel accumulates dQ over key tiles, both recomputing
//   P_ij = exp(E_ij - lambda log i - logZ_i), dR_ij = P_ij (dO_i . v_j - D_i),
//   dS_ij = dR_ij SiLU'(u_ij)  for j < i.
// No atomics: every output element is written by exactly one thread.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rel {
namespace simt {

constexpr int kRows = 64;     // query (or key) rows per CTA
constexpr int kTile = 64;     // rows per staged tile
constexpr int kThreads = 256; // 4 threads per row

template <typename TI>
struct IO;
template <>
struct IO<float> {
  static __device__ __forceinline__ float4 load4(const float* p) {
    return *reinterpret_cast<const float4*>(p);
  }
  static __device__ __forceinline__ void store4(float* p, float4 v) {
    *reinterpret_cast<float4*>(p) = v;
  }
};
template <>
struct IO<__nv_bfloat16> {
  static __device__ __forceinline__ float4 load4(const __nv_bfloat16* p) {
    uint2 raw = *reinterpret_cast<const uint2*>(p);
    __nv_bfloat162 a = *reinterpret_cast<__nv_bfloat162*>(&raw.x);
    __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162*>(&raw.y);
    float2 fa = __bfloat1622float2(a), fb = __bfloat1622float2(b);
    return make_float4(fa.x, fa.y, fb.x, fb.y);
  }
  static __device__ __forceinline__ void store4(__nv_bfloat16* p, float4 v) {
    __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y);
    __nv_bfloat162 b = __floats2bfloat162_rn(v.z, v.w);
    uint2 raw;
    raw.x = *reinterpret_cast<uint32_t*>(&a);
    raw.y = *reinterpret_cast<uint32_t*>(&b);
    *reinterpret_cast<uint2*>(p) = raw;
  }
};

__device__ __forceinline__ float sigmoidf_acc(float x) { return 1.0f / (1.0f + expf(-x)); }

// Thread `part` of a row group owns the float4 chunks part, part + 4, part + 8, ...
template <int D>
struct Chunks {
  static constexpr int N = D / 16;  // float4 chunks per thread
  static __device__ __forceinline__ int col(int part, int c) { return (part + 4 * c) * 4; }
};

template <typename TI, int D>
__device__ __forceinline__ void load_row_chunks(const TI* row, int part, float (&x)[D / 4]) {
#pragma unroll
  for (int c = 0; c < Chunks<D>::N; ++c) {
    float4 t = IO<TI>::load4(row + Chunks<D>::col(part, c));
    x[4 * c + 0] = t.x; x[4 * c + 1] = t.y; x[4 * c + 2] = t.z; x[4 * c + 3] = t.w;
  }
}

template <int D>
__device__ __forceinline__ float dot_part(const float (&x)[D / 4], const float* srow, int part) {
  float acc = 0.f;
#pragma unroll
  for (int c = 0; c < Chunks<D>::N; ++c) {
    float4 t = *reinterpret_cast<const float4*>(srow + Chunks<D>::col(part, c));
    acc = fmaf(x[4 * c + 0], t.x, acc);
    acc = fmaf(x[4 * c + 1], t.y, acc);
    acc = fmaf(x[4 * c + 2], t.z, acc);
    acc = fmaf(x[4 * c + 3], t.w, acc);
  }
  acc += __shfl_xor_sync(0xffffffffu, acc, 1);
  acc += __shfl_xor_sync(0xffffffffu, acc, 2);
  return acc;
}

template <int D>
__device__ __forceinline__ void axpy_part(float (&y)[D / 4], float a, const float* srow, int part) {
#pragma unroll
  for (int c = 0; c < Chunks<D>::N; ++c) {
    float4 t = *reinterpret_cast<const float4*>(srow + Chunks<D>::col(part, c));
    y[4 * c + 0] = fmaf(a, t.x, y[4 * c + 0]);
    y[4 * c + 1] = fmaf(a, t.y, y[4 * c + 1]);
    y[4 * c + 2] = fmaf(a, t.z, y[4 * c + 2]);
    y[4 * c + 3] = fmaf(a, t.w, y[4 * c + 3]);
  }
}

// Stage rows [r0, r0 + kTile) of one head of `src` into shared memory as fp32
// (rows >= T are zero).
template <typename TI, int D>
__device__ __forceinline__ void stage_tile(float* dst, const TI* src, long long sT, int r0, int T) {
  for (int idx = threadIdx.x; idx < kTile * (D / 4); idx += kThreads) {
    int rr = idx / (D / 4), c4 = idx % (D / 4);
    int r = r0 + rr;
    float4 t = make_float4(0.f, 0.f, 0.f, 0.f);
    if (r < T) t = IO<TI>::load4(src + (long long)r * sT + 4 * c4);
    *reinterpret_cast<float4*>(dst + rr * D + 4 * c4) = t;
  }
}

// ---------------------------------------------------------------------------
// Forward
// ---------------------------------------------------------------------------
template <typename TI, int D>
__global__ void __launch_bounds__(kThreads) fwd_kernel(Problem p) {
  extern __shared__ float4 smem_f4[];
  float* Ks = reinterpret_cast<float*>(smem_f4);
  float* Vs = Ks + kTile * D;
  const int rl = threadIdx.x >> 2, part = threadIdx.x & 3;
  const int bh = blockIdx.y, b = bh / p.H, h = bh % p.H;
  const int q0 = blockIdx.x * kRows;
  const int r = q0 + rl;
  const bool row_ok = r < p.T;
  const long long base = (long long)b * p.sB + (long long)h * p.sH;
  const TI* Q = reinterpret_cast<const TI*>(p.q) + base;
  const TI* K = reinterpret_cast<const TI*>(p.k) + base;
  const TI* V = reinterpret_cast<const TI*>(p.v) + base;

  float qv[D / 4], z[D / 4];
#pragma unroll
  for (int c = 0; c < D / 4; ++c) { qv[c] = 0.f; z[c] = 0.f; }
  if (row_ok) load_row_chunks<TI, D>(Q + (long long)r * p.sT, part, qv);

  float m = -INFINITY, l = 0.f, s_self = 0.f;
  const int kend = min(p.T, q0 + kRows);
  for (int k0 = 0; k0 < kend; k0 += kTile) {
    __syncthreads();
    stage_tile<TI, D>(Ks, K, p.sT, k0, p.T);
    stage_tile<TI, D>(Vs, V, p.sT, k0, p.T);
    __syncthreads();
    float e[kTile];
    float mt = -INFINITY;
#pragma unroll
    for (int jj = 0; jj < kTile; ++jj) {
      const float u = dot_part<D>(qv, Ks + jj * D, part) * p.inv_sqrt_d;
      const int j = k0 + jj;
      float ev = -INFINITY;
      if (j < r) {
        ev = u * sigmoidf_acc(u);                    // E_ij = SiLU(U_ij)
      } else if (j == r) {
        s_self = sigmoidf_acc(u / p.tau_s);          // S_i = sigmoid(U_ii / tau_S)
      }
      e[jj] = ev;
      mt = fmaxf(mt, ev);
    }
    const float mn = fmaxf(m, mt);
    if (mn == -INFINITY) continue;                   // no history seen yet
    const float sc = expf(m - mn);                   // e^{m - m'}; 0 for the empty state
    l *= sc;
#pragma unroll
    for (int c = 0; c < D / 4; ++c) z[c] *= sc;
#pragma unroll
    for (int jj = 0; jj < kTile; ++jj) {
      const float w = expf(e[jj] - mn);             // exp(-inf) = 0 outside the history
      l += w;
      axpy_part<D>(z, w, Vs + jj * D, part);
    }
    m = mn;
  }
  if (!row_ok) return;

  float g = 0.f, lz = s_self;
  float inv_l = 0.f, fself = 1.0f;  // F_ii = 1 - g: the Self flow
  if (r > 0 && l > 0.f) {
    const float A = m + logf(l) - p.lambda * logf((float)(r + 1));
    g = 1.0f / (1.0f + expf(s_self - A));
    fself = 1.0f / (1.0f + expf(A - s_self));
    const float hi = fmaxf(s_self, A), lo = fminf(s_self, A);
    lz = hi + log1pf(expf(lo - hi));
    inv_l = 1.0f / l;
  }
  float vi[D / 4];
  load_row_chunks<TI, D>(V + (long long)r * p.sT, part, vi);
  TI* Y = reinterpret_cast<TI*>(p.out) + base + (long long)r * p.sT;
#pragma unroll
  for (int c = 0; c < Chunks<D>::N; ++c) {
    float4 y;
    y.x = (1.f - g) * vi[4 * c + 0] + g * (z[4 * c + 0] * inv_l);
    y.y = (1.f - g) * vi[4 * c + 1] + g * (z[4 * c + 1] * inv_l);
    y.z = (1.f - g) * vi[4 * c + 2] + g * (z[4 * c + 2] * inv_l);
    y.w = (1.f - g) * vi[4 * c + 3] + g * (z[4 * c + 3] * inv_l);
    IO<TI>::store4(Y + Chunks<D>::col(part, c), y);
  }
  if (part == 0) {
    p.logz[(long long)bh * p.T + r] = lz;
    if (p.fself) p.fself[(long long)bh * p.T + r] = fself;
  }
}

// ---------------------------------------------------------------------------
// Backward: dK, dV (key-stationary)
// ---------------------------------------------------------------------------
template <typename TI, int D>
__global__ void __launch_bounds__(kThreads) bwd_dkdv_kernel(Problem p, BwdWorkspace ws) {
  extern __shared__ float4 smem_f4[];
  float* Qs = reinterpret_cast<float*>(smem_f4);
  float* Gs = Qs + kTile * D;        // dO tile
  float* cs = Gs + kTile * D;        // -lambda log i - logZ_i
  float* Ds = cs + kTile;            // D_i
  float* ws_l = Ds + kTile;          // log i * F_ii (Exchange weight of dlambda)
  __shared__ float red[kThreads / 32];
  const int rl = threadIdx.x >> 2, part = threadIdx.x & 3;
  const int bh = blockIdx.y, b = bh / p.H, h = bh % p.H;
  const int k0 = blockIdx.x * kRows;
  const int j = k0 + rl;
  const bool key_ok = j < p.T;
  const long long base = (long long)b * p.sB + (long long)h * p.sH;
  const TI* Q = reinterpret_cast<const TI*>(p.q) + base;
  const TI* K = reinterpret_cast<const TI*>(p.k) + base;
  const TI* V = reinterpret_cast<const TI*>(p.v) + base;
  const TI* G = reinterpret_cast<const TI*>(p.dout) + base;
  const float* logz = p.logz_in + (long long)bh * p.T;
  const float* Drow = ws.D + (long long)bh * p.T;

  float kv[D / 4], vv[D / 4], dk[D / 4], dv[D / 4];
#pragma unroll
  for (int c = 0; c < D / 4; ++c) { kv[c] = vv[c] = dk[c] = dv[c] = 0.f; }
  float dlam = 0.f;  // -sum_i log i F_ii dR_ij over this key's Exchange pairs
  if (key_ok) {
    load_row_chunks<TI, D>(K + (long long)j * p.sT, part, kv);
    load_row_chunks<TI, D>(V + (long long)j * p.sT, part, vv);
  }
  for (int q0 = k0; q0 < p.T; q0 += kTile) {
    __syncthreads();
    stage_tile<TI, D>(Qs, Q, p.sT, q0, p.T);
    stage_tile<TI, D>(Gs, G, p.sT, q0, p.T);
    for (int ii = threadIdx.x; ii < kTile; ii += kThreads) {
      const int i = q0 + ii;
      const float li = logf((float)(i + 1));
      cs[ii] = i < p.T ? -p.lambda * li - logz[i] : -INFINITY;
      Ds[ii] = i < p.T ? Drow[i] : 0.f;
      ws_l[ii] = i < p.T ? li * ws.F_self[(long long)bh * p.T + i] : 0.f;
    }
    __syncthreads();
    for (int ii = 0; ii < kTile; ++ii) {
      const int i = q0 + ii;
      const float u = dot_part<D>(kv, Qs + ii * D, part) * p.inv_sqrt_d;
      const float dP = dot_part<D>(vv, Gs + ii * D, part);
      if (i > j && i < p.T) {
        const float sg = sigmoidf_acc(u);
        const float E = u * sg;
        const float P = expf(E + cs[ii]);
        const float dR = P * (dP - Ds[ii]);
        const float dS = dR * (sg + E * (1.f - sg));   // SiLU'(u) = sigma + E (1 - sigma)
        dlam = fmaf(-ws_l[ii], dR, dlam);
        axpy_part<D>(dv, P, Gs + ii * D, part);
        axpy_part<D>(dk, dS, Qs + ii * D, part);
      }
    }
  }
  // per-CTA dlambda partial (the 4 threads of a key hold the same value: count part 0)
  float c = part == 0 ? dlam : 0.f;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) t += red[w];
    ws.dlam_part[ws.n_pre_blocks + blockIdx.y * gridDim.x + blockIdx.x] = t;
  }
  if (!key_ok) return;
  // Self terms of key j: dv_j += F_jj dO_j, dk_j += dS_jj q_j; then the 1/sqrt(d) of U.
  const long long row = (long long)bh * p.T + j;
  const float fs = ws.F_self[row], dss = ws.dS_self[row];
  float qj[D / 4], gj[D / 4];
  load_row_chunks<TI, D>(Q + (long long)j * p.sT, part, qj);
  load_row_chunks<TI, D>(G + (long long)j * p.sT, part, gj);
  TI* dK = reinterpret_cast<TI*>(p.dk) + base + (long long)j * p.sT;
  TI* dV = reinterpret_cast<TI*>(p.dv) + base + (long long)j * p.sT;
#pragma unroll
  for (int c = 0; c < Chunks<D>::N; ++c) {
    float4 a, v4;
    a.x = (dk[4 * c + 0] + dss * qj[4 * c + 0]) * p.inv_sqrt_d;
    a.y = (dk[4 * c + 1] + dss * qj[4 * c + 1]) * p.inv_sqrt_d;
    a.z = (dk[4 * c + 2] + dss * qj[4 * c + 2]) * p.inv_sqrt_d;
    a.w = (dk[4 * c + 3] + dss * qj[4 * c + 3]) * p.inv_sqrt_d;
    v4.x = dv[4 * c + 0] + fs * gj[4 * c + 0];
    v4.y = dv[4 * c + 1] + fs * gj[4 * c + 1];
    v4.z = dv[4 * c + 2] + fs * gj[4 * c + 2];
    v4.w = dv[4 * c + 3] + fs * gj[4 * c + 3];
    IO<TI>::store4(dK + Chunks<D>::col(part, c), a);
    IO<TI>::store4(dV + Chunks<D>::col(part, c), v4);
  }
}

// ---------------------------------------------------------------------------
// Backward: dQ (query-stationary)
// ---------------------------------------------------------------------------
template <typename TI, int D>
__global__ void __launch_bounds__(kThreads) bwd_dq_kernel(Problem p, BwdWorkspace ws) {
  extern __shared__ float4 smem_f4[];
  float* Ks = reinterpret_cast<float*>(smem_f4);
  float* Vs = Ks + kTile * D;
  const int rl = threadIdx.x >> 2, part = threadIdx.x & 3;
  const int bh = blockIdx.y, b = bh / p.H, h = bh % p.H;
  const int q0 = blockIdx.x * kRows;
  const int i = q0 + rl;
  const bool row_ok = i < p.T;
  const long long base = (long long)b * p.sB + (long long)h * p.sH;
  const TI* Q = reinterpret_cast<const TI*>(p.q) + base;
  const TI* K = reinterpret_cast<const TI*>(p.k) + base;
  const TI* V = reinterpret_cast<const TI*>(p.v) + base;
  const TI* G = reinterpret_cast<const TI*>(p.dout) + base;
  const long long row = (long long)bh * p.T + i;

  float qv[D / 4], gv[D / 4], dq[D / 4];
#pragma unroll
  for (int c = 0; c < D / 4; ++c) { qv[c] = gv[c] = dq[c] = 0.f; }
  float ci = -INFINITY, Di = 0.f;
  if (row_ok) {
    load_row_chunks<TI, D>(Q + (long long)i * p.sT, part, qv);
    load_row_chunks<TI, D>(G + (long long)i * p.sT, part, gv);
    ci = -p.lambda * logf((float)(i + 1)) - p.logz_in[row];
    Di = ws.D[row];
  }
  const int kend = min(p.T, q0 + kRows);
  for (int k0 = 0; k0 < kend; k0 += kTile) {
    __syncthreads();
    stage_tile<TI, D>(Ks, K, p.sT, k0, p.T);
    stage_tile<TI, D>(Vs, V, p.sT, k0, p.T);
    __syncthreads();
    for (int jj = 0; jj < kTile; ++jj) {
      const int j = k0 + jj;
      const float u = dot_part<D>(qv, Ks + jj * D, part) * p.inv_sqrt_d;
      const float dP = dot_part<D>(gv, Vs + jj * D, part);
      if (j < i && row_ok) {
        const float sg = sigmoidf_acc(u);
        const float E = u * sg;
        const float P = expf(E + ci);
        const float dR = P * (dP - Di);
        const float dS = dR * (sg + E * (1.f - sg));
        axpy_part<D>(dq, dS, Ks + jj * D, part);
      }
    }
  }
  if (!row_ok) return;
  const float dss = ws.dS_self[row];
  float ki[D / 4];
  load_row_chunks<TI, D>(K + (long long)i * p.sT, part, ki);
  TI* dQ = reinterpret_cast<TI*>(p.dq) + base + (long long)i * p.sT;
#pragma unroll
  for (int c = 0; c < Chunks<D>::N; ++c) {
    float4 a;
    a.x = (dq[4 * c + 0] + dss * ki[4 * c + 0]) * p.inv_sqrt_d;
    a.y = (dq[4 * c + 1] + dss * ki[4 * c + 1]) * p.inv_sqrt_d;
    a.z = (dq[4 * c + 2] + dss * ki[4 * c + 2]) * p.inv_sqrt_d;
    a.w = (dq[4 * c + 3] + dss * ki[4 * c + 3]) * p.inv_sqrt_d;
    IO<TI>::store4(dQ + Chunks<D>::col(part, c), a);
  }
}

// ---------------------------------------------------------------------------
// Launchers
// ---------------------------------------------------------------------------
bool supports(relation_dtype dt, int d) {
  (void)dt;
  return d == 32 || d == 64 || d == 128;
}

template <typename TI, int D>
static cudaError_t fwd_t(const Problem& p, cudaStream_t s) {
  const size_t smem = 2u * kTile * D * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(fwd_kernel<TI, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((p.T + kRows - 1) / kRows, p.B * p.H);
  fwd_kernel<TI, D><<<grid, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <typename TI, int D>
static cudaError_t bwd_t(const Problem& p, const BwdWorkspace& ws, cudaStream_t s) {
  const size_t smem_kv = 2u * kTile * D * sizeof(float) + 3u * kTile * sizeof(float);
  const size_t smem_q = 2u * kTile * D * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(bwd_dkdv_kernel<TI, D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_kv);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(bwd_dq_kernel<TI, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem_q);
  if (e != cudaSuccess) return e;
  dim3 grid((p.T + kRows - 1) / kRows, p.B * p.H);
  bwd_dkdv_kernel<TI, D><<<grid, kThreads, smem_kv, s>>>(p, ws);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  bwd_dq_kernel<TI, D><<<grid, kThreads, smem_q, s>>>(p, ws);
  return cudaGetLastError();
}

int main_ctas(const Problem& p) { return ((p.T + kRows - 1) / kRows) * p.B * p.H; }

cudaError_t launch_fwd(const Problem& p, cudaStream_t s) {
  if (p.dtype == RELATION_F32) {
    switch (p.d) {
      case 32: return fwd_t<float, 32>(p, s);
      case 64: return fwd_t<float, 64>(p, s);
      case 128: return fwd_t<float, 128>(p, s);
    }
  } else {
    switch (p.d) {
      case 32: return fwd_t<__nv_bfloat16, 32>(p, s);
      case 64: return fwd_t<__nv_bfloat16, 64>(p, s);
      case 128: return fwd_t<__nv_bfloat16, 128>(p, s);
    }
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_bwd(const Problem& p, const BwdWorkspace& ws, cudaStream_t s) {
  if (p.dtype == RELATION_F32) {
    switch (p.d) {
      case 32: return bwd_t<float, 32>(p, ws, s);
      case 64: return bwd_t<float, 64>(p, ws, s);
      case 128: return bwd_t<float, 128>(p, ws, s);
    }
  } else {
    switch (p.d) {
      case 32: return bwd_t<__nv_bfloat16, 32>(p, ws, s);
      case 64: return bwd_t<__nv_bfloat16, 64>(p, ws, s);
      case 128: return bwd_t<__nv_bfloat16, 128>(p, ws, s);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace simt
}  // namespace rel
