// relation_linear.cu -- Linear Relation (Sec. 5.2, App. A.4): the recurrent Exchange form.
//
// Per head, tokens t = 1..T, state C in R^{d x d} (rows on the coordinate side, columns on
// the information side), C_0 = 0:
//   Ask Self:     S_t = sigmoid(p1_t . p2_t / (tau_S sqrt d)),  ^p = p / |p|
//   Ask Others:   C^- = Diag(alpha_t) C_{t-1},  E_t = S_t (C^-)^T ^p1_t
//   Answer:       Y_t = I~_t + E_t
//   Become Others: C_t = C^- + S_t ^p2_t I~_t^T
// alpha_t in (0, 1]^d is the channel-wise retention (an input; its KDA parameterisation
// of Eq. (retention-vector) is upstream), p1, p2 are taken after RoPE (upstream).
//
// The recurrence never mixes information columns: column j of C evolves on its own.  The
// forward therefore gives thread (j, half) column j for half of the rows, with that part
// of the state in registers; a token costs d/2 multiply-adds three times per thread and
// one pair shuffle (the two halves of the read).  One CTA per (b, h) walks the tokens in
// order; tokens are staged through shared memory in chunks of kChunkT, double-buffered,
// with S_t, 1/|p1_t|, 1/|p2_t| computed per chunk (S is folded into the coordinates:
// q'_t = S_t ^p1_t, k'_t = S_t ^p2_t).
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rel {
namespace lin {

constexpr int kChunkT = 16;  // tokens per staged chunk

template <typename TI>
__device__ __forceinline__ float ldx(const TI* p);
template <>
__device__ __forceinline__ float ldx<float>(const float* p) { return *p; }
template <>
__device__ __forceinline__ float ldx<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}
template <typename TI>
__device__ __forceinline__ void stx(TI* p, float v);
template <>
__device__ __forceinline__ void stx<float>(float* p, float v) { *p = v; }
template <>
__device__ __forceinline__ void stx<__nv_bfloat16>(__nv_bfloat16* p, float v) {
  *p = __float2bfloat16_rn(v);
}

// Shared staging of one chunk: per token the four vectors alpha, q', k', I~ (fp32).
template <int D>
struct Chunk {
  float vec[kChunkT][4][D];  // [0] alpha, [1] p1 -> q', [2] p2 -> k', [3] I~
  float scal[kChunkT][4];    // S, 1/|p1|, 1/|p2|
};

// Raw loads of chunk `ch` (tokens ch * kChunkT ...) into registers: element e of the
// chunk's 4 * kChunkT * D values goes to thread e % NT, slot e / NT.
template <typename TI, int D, int NT>
struct Loader {
  static constexpr int N = 4 * kChunkT * D / NT;  // values per thread
  float r[N];
  __device__ __forceinline__ void load(const LinearProblem& p, int b, int h, int ch) {
#pragma unroll
    for (int n = 0; n < N; ++n) {
      const int e = n * NT + (int)threadIdx.x;
      const int c = e % D, a = (e / D) % 4, tt = e / (4 * D);
      const int t = ch * kChunkT + tt;
      float x = 0.f;
      if (t < p.T) {
        const long long off = (long long)b * p.sB + (long long)t * p.sT + (long long)h * p.sH + c;
        if (a == 0) x = p.alpha[off];
        else if (a == 1) x = ldx<TI>(reinterpret_cast<const TI*>(p.p1) + off);
        else if (a == 2) x = ldx<TI>(reinterpret_cast<const TI*>(p.p2) + off);
        else x = ldx<TI>(reinterpret_cast<const TI*>(p.v) + off);
      }
      r[n] = x;
    }
  }
  __device__ __forceinline__ void store(Chunk<D>& s) const {
#pragma unroll
    for (int n = 0; n < N; ++n) {
      const int e = n * NT + (int)threadIdx.x;
      (&s.vec[0][0][0])[e] = r[n];
    }
  }
};

// Ask Self for the chunk's tokens (one warp per token), then fold S into the unit
// coordinates.  Two block barriers; the caller has made the raw values visible.
template <int D, int NT>
__device__ __forceinline__ void ask_self_chunk(Chunk<D>& s, float tau_s) {
  constexpr int NW = NT / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int tt = warp; tt < kChunkT; tt += NW) {
    float s12 = 0.f, s11 = 0.f, s22 = 0.f;
    for (int c = lane; c < D; c += 32) {
      const float a = s.vec[tt][1][c], b = s.vec[tt][2][c];
      s12 = fmaf(a, b, s12);
      s11 = fmaf(a, a, s11);
      s22 = fmaf(b, b, s22);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      s12 += __shfl_xor_sync(0xffffffffu, s12, o);
      s11 += __shfl_xor_sync(0xffffffffu, s11, o);
      s22 += __shfl_xor_sync(0xffffffffu, s22, o);
    }
    if (lane == 0) {
      s.scal[tt][0] = 1.0f / (1.0f + expf(-s12 / (tau_s * sqrtf((float)D))));
      s.scal[tt][1] = s11 > 0.f ? rsqrtf(s11) : 0.f;
      s.scal[tt][2] = s22 > 0.f ? rsqrtf(s22) : 0.f;
    }
  }
  __syncthreads();
  for (int e = threadIdx.x; e < kChunkT * 2 * D; e += NT) {
    const int c = e % D, a = 1 + (e / D) % 2, tt = e / (2 * D);
    s.vec[tt][a][c] *= s.scal[tt][0] * s.scal[tt][a];
  }
  __syncthreads();
}

// Forward: one CTA per head, thread (j, half) = column j, rows half * D/2 .. + D/2.
template <typename TI, int D>
__global__ void __launch_bounds__(2 * D) fwd_kernel(LinearProblem p) {
  constexpr int NT = 2 * D, R = D / 2;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  Chunk<D>* buf = reinterpret_cast<Chunk<D>*>(smem_raw);
  const int bh = blockIdx.x, b = bh / p.H, h = bh % p.H;
  const int j = threadIdx.x >> 1, half = threadIdx.x & 1, r0 = half * R;
  const int n_ch = (p.T + kChunkT - 1) / kChunkT;
  float C[R];
#pragma unroll
  for (int r = 0; r < R; ++r) C[r] = 0.f;
  Loader<TI, D, NT> ld;
  ld.load(p, b, h, 0);
  ld.store(buf[0]);
  __syncthreads();
  ask_self_chunk<D, NT>(buf[0], p.tau_s);
  TI* Y = reinterpret_cast<TI*>(p.y) + (long long)b * p.sB + (long long)h * p.sH + j;
  for (int ch = 0; ch < n_ch; ++ch) {
    Chunk<D>& cur = buf[ch & 1];
    const bool more = ch + 1 < n_ch;
    if (more) ld.load(p, b, h, ch + 1);  // in flight while this chunk is computed
    const int nt = min(kChunkT, p.T - ch * kChunkT);
    for (int tt = 0; tt < nt; ++tt) {
      const float* al = &cur.vec[tt][0][r0];
      const float* qp = &cur.vec[tt][1][r0];
      const float* kp = &cur.vec[tt][2][r0];
      const float I = cur.vec[tt][3][j];
      float e = 0.f;
#pragma unroll
      for (int r = 0; r < R; r += 4) {
        const float4 a4 = *reinterpret_cast<const float4*>(al + r);
        const float4 q4 = *reinterpret_cast<const float4*>(qp + r);
        const float4 k4 = *reinterpret_cast<const float4*>(kp + r);
        const float av[4] = {a4.x, a4.y, a4.z, a4.w}, qv[4] = {q4.x, q4.y, q4.z, q4.w};
        const float kv[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float cm = C[r + u] * av[u];  // Ask Others: decayed state
          e = fmaf(cm, qv[u], e);              // read with S q^
          C[r + u] = fmaf(kv[u], I, cm);       // Become Others: write S k^ I~
        }
      }
      e += __shfl_xor_sync(0xffffffffu, e, 1);  // the other half of the rows
      if (half == 0) stx<TI>(Y + (long long)(ch * kChunkT + tt) * p.sT, I + e);  // Answer
    }
    if (more) {
      // nxt held chunk ch - 1, which every thread finished before the barriers that ended
      // the previous iteration
      Chunk<D>& nxt = buf[(ch + 1) & 1];
      ld.store(nxt);
      __syncthreads();
      ask_self_chunk<D, NT>(nxt, p.tau_s);
    }
  }
}

template <typename TI, int D>
cudaError_t fwd_t(const LinearProblem& p, cudaStream_t s) {
  const int smem = 2 * (int)sizeof(Chunk<D>);
  cudaError_t e = cudaFuncSetAttribute(fwd_kernel<TI, D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) { note_failure("linear forward: shared memory attribute"); return e; }
  fwd_kernel<TI, D><<<(unsigned)(p.B * p.H), 2 * D, smem, s>>>(p);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("linear forward: launch");
  return e;
}

}  // namespace lin

bool linear_supports(relation_dtype dt, int d) {
  return (dt == RELATION_F32 || dt == RELATION_BF16) && (d == 32 || d == 64);
}

cudaError_t launch_linear_fwd(const LinearProblem& p, cudaStream_t s) {
  if (p.dtype == RELATION_F32)
    return p.d == 32 ? lin::fwd_t<float, 32>(p, s) : lin::fwd_t<float, 64>(p, s);
  return p.d == 32 ? lin::fwd_t<__nv_bfloat16, 32>(p, s) : lin::fwd_t<__nv_bfloat16, 64>(p, s);
}

}  // namespace rel
