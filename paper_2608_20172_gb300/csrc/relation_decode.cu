// relation_decode.cu -- one new token per sequence against a key/value cache.
//
// Decoding with the causal Relation operator (Sec. 3.1; the factorised row of Sec. 4.2 /
// App. A.1): sequence b of the batch holds len_b cached rows whose last row is the new
// token, at one-based position i = len_b.  Per (b, h):
//   Exchange over the history j < i (cache rows 0 .. len_b - 2):
//       E_j = SiLU(q . k_j / sqrt(d)),  L^E = log sum_j e^{E_j},  z = sum_j e^{E_j} v_j
//   Self (cache row len_b - 1):  S = sigmoid(q . k_i / (sqrt(d) tau_S))
//   A = L^E - lambda log i,  g = sigmoid(A - S),  Y = (1 - g) v_i + g z / sum_j e^{E_j},
//   logZ = logaddexp(S, A);  a one-row cache (i = 1) has no history: g = 0, Y = v_1,
//   logZ = S.
// This is the last row of the full forward over the cache, evaluated without the other
// rows.  Memory-bound: every cached key and value is read once.
//
// Two launches.  The partial pass splits each history into chunks of kChunk rows, one CTA
// per (head, chunk): 8 warps take the chunk's rows in turn (scores with four lanes per
// key, P V with the lanes spanning d), and the CTA leaves (m, l, z) = (max E, sum e^{E - m}, sum e^{E - m} v) in the
// workspace.  The combine pass (one CTA per head, one thread per column) merges the
// chunks with the associative (m, l, z) rule of the tiled scan (App. A.3) and applies the
// Self-Exchange epilogue.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rel {
namespace decode {

constexpr int kChunk = 512;   // history rows per partial CTA
constexpr int kWarps = 8;
constexpr int kMaxD = 128;

template <typename TI>
__device__ __forceinline__ float ldf(const TI* p);
template <>
__device__ __forceinline__ float ldf<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float ldf<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}

// Loads of n consecutive elements as fp32 (n * sizeof(TI) is 4, 8 or 16 bytes, aligned).
template <typename TI, int N>
__device__ __forceinline__ void ld_vec(const TI* p, float* out) {
  if constexpr (sizeof(TI) == 4) {
    static_assert(N % 4 == 0 || N <= 2, "fp32 vector width");
    if constexpr (N == 1) {
      out[0] = __ldg(reinterpret_cast<const float*>(p));
    } else if constexpr (N == 2) {
      const float2 v = __ldg(reinterpret_cast<const float2*>(p));
      out[0] = v.x; out[1] = v.y;
    } else {
#pragma unroll
      for (int i = 0; i < N; i += 4) {
        const float4 v = __ldg(reinterpret_cast<const float4*>(p + i));
        out[i] = v.x; out[i + 1] = v.y; out[i + 2] = v.z; out[i + 3] = v.w;
      }
    }
  } else {
    if constexpr (N == 2) {
      const uint32_t w = __ldg(reinterpret_cast<const unsigned int*>(p));
      const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w));
      out[0] = f.x; out[1] = f.y;
    } else if constexpr (N == 4) {
      const uint2 w = __ldg(reinterpret_cast<const uint2*>(p));
      const uint32_t ww[2] = {w.x, w.y};
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ww[e]));
        out[2 * e] = f.x; out[2 * e + 1] = f.y;
      }
    } else {
      static_assert(N % 8 == 0, "bf16 vector width");
#pragma unroll
      for (int i = 0; i < N; i += 8) {
        const uint4 w = __ldg(reinterpret_cast<const uint4*>(p + i));
        const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ww[e]));
          out[i + 2 * e] = f.x; out[i + 2 * e + 1] = f.y;
        }
      }
    }
  }
}

// Partial (m, l, z) of history rows [c0, min(c0 + kChunk, len - 1)) of head (b, h).
// D = 64 or 128: vector loads (scores: four lanes per key, each a quarter of the row;
// P V: each lane D / 32 consecutive columns).  D = 0: any d_h <= 128, one element per
// lane per load.
template <typename TI, int D>
__global__ void __launch_bounds__(kWarps * 32) partial_kernel(DecodeProblem p, float* part) {
  __shared__ float e_s[kChunk];
  __shared__ float red[kWarps];
  __shared__ float zs[kWarps][kMaxD];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.x, chunk = blockIdx.y;
  const int b = bh / p.H, h = bh % p.H;
  const int len = p.lengths[b];
  if (len < 1 || len > p.T) {  // invalid length: report it, touch no cache row
    if (threadIdx.x == 0 && chunk == 0 && p.dev_status)
      atomicExch(p.dev_status, (int)RELATION_ERR_INVALID_ARG);
    return;
  }
  const int hist = len - 1;  // history rows
  const int c0 = chunk * kChunk;
  const int n = max(0, min(kChunk, hist - c0));
  const TI* qv = reinterpret_cast<const TI*>(p.q) + (long long)b * p.qsB + (long long)h * p.qsH;
  const TI* kc = reinterpret_cast<const TI*>(p.k) + (long long)b * p.sB + (long long)h * p.sH +
                 (long long)c0 * p.sT;
  const TI* vc = reinterpret_cast<const TI*>(p.v) + (long long)b * p.sB + (long long)h * p.sH +
                 (long long)c0 * p.sT;
  constexpr int PL = D > 0 ? D / 32 : kMaxD / 32;  // columns per lane in the P V pass
  float mx = -INFINITY;
  if constexpr (D > 0) {
    // scores: lane = 4 key + quarter; per iteration two groups of 8 keys,
    // jj = base + lane / 4 and jj + 8 kWarps, loaded together (rows past the chunk read a
    // clamped row and are dropped)
    constexpr int QD = D / 4;
    const int sub = lane & 3, slot = lane >> 2;
    float qr[QD];
    ld_vec<TI, QD>(qv + sub * QD, qr);
    for (int base = warp * 8; base < n; base += 16 * kWarps) {
      const int j0 = base + slot, j1 = j0 + 8 * kWarps;
      float k0[QD], k1[QD];
      ld_vec<TI, QD>(kc + (long long)min(j0, n - 1) * p.sT + sub * QD, k0);
      ld_vec<TI, QD>(kc + (long long)min(j1, n - 1) * p.sT + sub * QD, k1);
      float s0 = 0.f, s1 = 0.f;
#pragma unroll
      for (int e = 0; e < QD; ++e) {
        s0 = fmaf(qr[e], k0[e], s0);
        s1 = fmaf(qr[e], k1[e], s1);
      }
      s0 += __shfl_xor_sync(0xffffffffu, s0, 1);
      s1 += __shfl_xor_sync(0xffffffffu, s1, 1);
      s0 += __shfl_xor_sync(0xffffffffu, s0, 2);
      s1 += __shfl_xor_sync(0xffffffffu, s1, 2);
      if (j0 < n) {
        const float u = s0 * p.inv_sqrt_d;
        const float E = u / (1.0f + expf(-u));  // SiLU(u)
        if (sub == 0) e_s[j0] = E;
        mx = fmaxf(mx, E);
      }
      if (j1 < n) {
        const float u = s1 * p.inv_sqrt_d;
        const float E = u / (1.0f + expf(-u));
        if (sub == 0) e_s[j1] = E;
        mx = fmaxf(mx, E);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  } else {
    float qr[PL];
#pragma unroll
    for (int e = 0; e < PL; ++e) {
      const int c = lane + 32 * e;
      qr[e] = c < p.d ? ldf<TI>(qv + c) : 0.f;
    }
    for (int jj = warp; jj < n; jj += kWarps) {
      const TI* kr = kc + (long long)jj * p.sT;
      float s = 0.f;
#pragma unroll
      for (int e = 0; e < PL; ++e) {
        const int c = lane + 32 * e;
        if (c < p.d) s = fmaf(qr[e], ldf<TI>(kr + c), s);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      const float u = s * p.inv_sqrt_d;
      const float E = u / (1.0f + expf(-u));  // SiLU(u)
      if (lane == 0) e_s[jj] = E;
      mx = fmaxf(mx, E);
    }
  }
  if (lane == 0) red[warp] = mx;
  __syncthreads();
  float m = -INFINITY;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) m = fmaxf(m, red[w]);
  __syncthreads();
  // l = sum e^{E - m},  z = sum e^{E - m} v_j
  float l = 0.f, z[PL];
#pragma unroll
  for (int e = 0; e < PL; ++e) z[e] = 0.f;
  if constexpr (D > 0) {
    const int col = lane * PL;
#pragma unroll 8
    for (int jj = warp; jj < n; jj += kWarps) {
      const float P = expf(e_s[jj] - m);
      l += P;
      float vr[PL];
      ld_vec<TI, PL>(vc + (long long)jj * p.sT + col, vr);
#pragma unroll
      for (int e = 0; e < PL; ++e) z[e] = fmaf(P, vr[e], z[e]);
    }
#pragma unroll
    for (int e = 0; e < PL; ++e) zs[warp][col + e] = z[e];
  } else {
    for (int jj = warp; jj < n; jj += kWarps) {
      const float P = expf(e_s[jj] - m);
      l += P;
      const TI* vr = vc + (long long)jj * p.sT;
#pragma unroll
      for (int e = 0; e < PL; ++e) {
        const int c = lane + 32 * e;
        if (c < p.d) z[e] = fmaf(P, ldf<TI>(vr + c), z[e]);
      }
    }
#pragma unroll
    for (int e = 0; e < PL; ++e) zs[warp][lane + 32 * e] = z[e];
  }
  if (lane == 0) red[warp] = l;
  __syncthreads();
  float* out = part + ((long long)bh * gridDim.y + chunk) * (2 + kMaxD);
  if (threadIdx.x == 0) {
    float lt = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) lt += red[w];
    out[0] = m;   // -inf for an empty chunk
    out[1] = lt;  // 0 for an empty chunk
  }
  for (int c = threadIdx.x; c < p.d; c += blockDim.x) {
    float zt = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) zt += zs[w][c];
    out[2 + c] = zt;
  }
}

// Merge the chunks of head (b, h) and apply the Self-Exchange epilogue; thread c owns
// column c (blockDim.x = kMaxD, threads c >= d only join the reductions).
template <typename TI>
__global__ void __launch_bounds__(kMaxD) combine_kernel(DecodeProblem p, const float* part,
                                                        int n_chunks) {
  __shared__ float red[kMaxD / 32];
  const int bh = blockIdx.x, c = threadIdx.x;
  const int b = bh / p.H, h = bh % p.H;
  const int len = p.lengths[b];
  if (len < 1 || len > p.T) return;  // reported by the partial pass
  const int lane = c & 31, warp = c >> 5;
  const TI* qv = reinterpret_cast<const TI*>(p.q) + (long long)b * p.qsB + (long long)h * p.qsH;
  const long long self_row = (long long)b * p.sB + (long long)h * p.sH + (long long)(len - 1) * p.sT;
  const TI* ks = reinterpret_cast<const TI*>(p.k) + self_row;
  const TI* vs = reinterpret_cast<const TI*>(p.v) + self_row;
  // Self evidence q . k_i
  float s = c < p.d ? ldf<TI>(qv + c) * ldf<TI>(ks + c) : 0.f;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) red[warp] = s;
  __syncthreads();
  float qk = 0.f;
#pragma unroll
  for (int w = 0; w < kMaxD / 32; ++w) qk += red[w];
  const float S = 1.0f / (1.0f + expf(-(qk * p.inv_sqrt_d) / p.tau_s));
  // (m, l, z) merge over the chunks that hold history
  const int used = (len - 1 + kChunk - 1) / kChunk;  // <= n_chunks
  const float* pb = part + (long long)bh * n_chunks * (2 + kMaxD);
  float M = -INFINITY;
  for (int k = 0; k < used; ++k) M = fmaxf(M, pb[k * (2 + kMaxD)]);
  float L = 0.f, Z = 0.f;
  for (int k = 0; k < used; ++k) {
    const float* pk = pb + k * (2 + kMaxD);
    const float w = pk[0] == -INFINITY ? 0.f : expf(pk[0] - M);
    L = fmaf(w, pk[1], L);
    if (c < p.d) Z = fmaf(w, pk[2 + c], Z);
  }
  float g = 0.f, lz = S, fz = 0.f;
  if (len > 1 && L > 0.f) {
    const float A = M + logf(L) - p.lambda * logf((float)len);
    g = 1.0f / (1.0f + expf(S - A));
    const float hi = fmaxf(S, A), lo = fminf(S, A);
    lz = hi + log1pf(expf(lo - hi));
    fz = Z / L;
  }
  if (c < p.d) {
    const float vi = ldf<TI>(vs + c);
    const float y = fmaf(g, fz - vi, vi);
    TI* o = reinterpret_cast<TI*>(p.out) + (long long)b * p.qsB + (long long)h * p.qsH;
    if (sizeof(TI) == 4)
      reinterpret_cast<float*>(o)[c] = y;
    else
      reinterpret_cast<__nv_bfloat16*>(o)[c] = __float2bfloat16_rn(y);
  }
  if (c == 0) p.logz[bh] = lz;
}

template <typename TI>
cudaError_t launch_t(const DecodeProblem& p, float* part, int n_chunks, cudaStream_t s) {
  const dim3 grid((unsigned)(p.B * p.H), (unsigned)n_chunks);
  // vector loads need 16-byte aligned rows (strides are multiples of 16 bytes) and q
  const bool qal = (reinterpret_cast<uintptr_t>(p.q) & 15u) == 0 &&
                   (p.qsB * (long long)sizeof(TI)) % 16 == 0 &&
                   (p.qsH * (long long)sizeof(TI)) % 16 == 0;
  const bool kal = (p.sB * (long long)sizeof(TI)) % 16 == 0 &&
                   (p.sT * (long long)sizeof(TI)) % 16 == 0 &&
                   (p.sH * (long long)sizeof(TI)) % 16 == 0;
  if (qal && kal && p.d == 128)
    partial_kernel<TI, 128><<<grid, kWarps * 32, 0, s>>>(p, part);
  else if (qal && kal && p.d == 64)
    partial_kernel<TI, 64><<<grid, kWarps * 32, 0, s>>>(p, part);
  else
    partial_kernel<TI, 0><<<grid, kWarps * 32, 0, s>>>(p, part);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { note_failure("decode: partial pass launch"); return e; }
  combine_kernel<TI><<<(unsigned)(p.B * p.H), kMaxD, 0, s>>>(p, part, n_chunks);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("decode: combine launch");
  return e;
}

}  // namespace decode

int decode_chunks(int t_max) { return t_max > 1 ? (t_max - 1 + decode::kChunk - 1) / decode::kChunk : 1; }

size_t decode_workspace_bytes(int B, int H, int t_max) {
  return (size_t)B * H * decode_chunks(t_max) * (2 + decode::kMaxD) * sizeof(float);
}

cudaError_t launch_decode(const DecodeProblem& p, void* workspace, cudaStream_t s) {
  float* part = static_cast<float*>(workspace);
  const int n = decode_chunks(p.T);
  if (p.dtype == RELATION_F32) return decode::launch_t<float>(p, part, n, s);
  return decode::launch_t<__nv_bfloat16>(p, part, n, s);
}

}  // namespace rel
