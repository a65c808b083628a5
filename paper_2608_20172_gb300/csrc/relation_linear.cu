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
// forward therefore gives each column to kRG threads, each keeping d / kRG rows of it in
// registers; a token costs 3 d / kRG multiply-adds per thread (the read is summed over
// the column's threads once per chunk).  One CTA per (b, h) walks the tokens in
// order; tokens are staged through shared memory in double-buffered chunks, with S_t,
// 1/|p1_t|, 1/|p2_t| computed per chunk (S is folded into the coordinates:
// q'_t = S_t ^p1_t, k'_t = S_t ^p2_t).  Loads are 4-element vectors without conditions.
// The backward (below) walks the tokens in reverse with the adjoint state, recomputing
// the states of each chunk of kChunkB tokens from checkpoints the kernel stores first.
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

// Shared staging of one chunk of NTOK tokens: per token the four vectors alpha, q', k',
// I~ (fp32).
template <int D, int NTOK = kChunkT>
struct Chunk {
  float vec[NTOK][4][D];  // [0] alpha, [1] p1 -> q', [2] p2 -> k', [3] I~
  float scal[NTOK][4];    // S, 1/|p1|, 1/|p2|
};

// Four consecutive elements as fp32 (8- or 16-byte aligned vector load).
template <typename TI>
__device__ __forceinline__ float4 ld4(const TI* p);
template <>
__device__ __forceinline__ float4 ld4<float>(const float* p) {
  return *reinterpret_cast<const float4*>(p);
}
template <>
__device__ __forceinline__ float4 ld4<__nv_bfloat16>(const __nv_bfloat16* p) {
  const uint2 w = *reinterpret_cast<const uint2*>(p);
  const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w.x));
  const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w.y));
  return make_float4(lo.x, lo.y, hi.x, hi.y);
}

// Loads of chunk `ch` (tokens ch * NTOK ...) into registers as 4-element vectors: vector
// v of an array (token v / (D/4), columns 4 (v % (D/4)) ..) goes to thread v % NT.  The
// loads carry no condition (rows past T are clamped to T - 1 and zeroed after the load),
// so a thread's loads are all in flight together.
template <typename TI, int D, int NT, int NTOK = kChunkT>
struct Loader {
  static constexpr int NV = NTOK * D / 4 / NT;  // vectors per thread and array
  static_assert(NV >= 1 && NV * NT * 4 == NTOK * D, "chunk / thread split");
  float4 r[4][NV];
  __device__ __forceinline__ void load(const LinearProblem& p, int b, int h, int ch) {
#pragma unroll
    for (int n = 0; n < NV; ++n) {
      const int v = n * NT + (int)threadIdx.x;
      const int tt = v / (D / 4), c4 = (v % (D / 4)) * 4;
      const int t = ch * NTOK + tt, tc = min(t, p.T - 1);
      const long long off =
          (long long)b * p.sB + (long long)tc * p.sT + (long long)h * p.sH + c4;
      float4 x[4];
      x[0] = ld4<float>(p.alpha + off);
      x[1] = ld4<TI>(reinterpret_cast<const TI*>(p.p1) + off);
      x[2] = ld4<TI>(reinterpret_cast<const TI*>(p.p2) + off);
      x[3] = ld4<TI>(reinterpret_cast<const TI*>(p.v) + off);
#pragma unroll
      for (int a = 0; a < 4; ++a) r[a][n] = t < p.T ? x[a] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  __device__ __forceinline__ void store(Chunk<D, NTOK>& s) const {
#pragma unroll
    for (int n = 0; n < NV; ++n) {
      const int v = n * NT + (int)threadIdx.x;
      const int tt = v / (D / 4), c4 = (v % (D / 4)) * 4;
#pragma unroll
      for (int a = 0; a < 4; ++a) *reinterpret_cast<float4*>(&s.vec[tt][a][c4]) = r[a][n];
    }
  }
};

// Ask Self for the chunk's tokens (one warp per token), then fold S into the unit
// coordinates.  Two block barriers; the caller has made the raw values visible.
template <int D, int NT, int NTOK = kChunkT>
__device__ __forceinline__ void ask_self_chunk(Chunk<D, NTOK>& s, float tau_s) {
  constexpr int NW = NT / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int tt = warp; tt < NTOK; tt += NW) {
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
  for (int e = threadIdx.x; e < NTOK * 2 * D; e += NT) {
    const int c = e % D, a = 1 + (e / D) % 2, tt = e / (2 * D);
    s.vec[tt][a][c] *= s.scal[tt][0] * s.scal[tt][a];
  }
  __syncthreads();
}

// Forward: one CTA per head, kRG threads per column.  Thread (j, rg) = tid % D, tid / D
// keeps rows rg * D/kRG .. + D/kRG of column j in registers.  A warp shares one row group,
// so the per-token alpha, q', k' reads are one shared-memory broadcast per vector, and
// each thread's partial read goes to shared memory: Y_t = I~_t + sum_rg e_rg is formed per
// chunk (the output does not feed back into the recurrence), with no per-token shuffle.
constexpr int kRG = 4;
constexpr int kChunkF = 32;  // tokens per staged chunk (forward)

template <int D>
struct FwdSmem {
  Chunk<D, kChunkF> buf[2];
  float epart[kChunkF][kRG][D];  // partial reads of the chunk's tokens
};

template <typename TI, int D>
__global__ void __launch_bounds__(kRG * D) fwd_kernel(LinearProblem p) {
  constexpr int NT = kRG * D, R = D / kRG;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  FwdSmem<D>& sm = *reinterpret_cast<FwdSmem<D>*>(smem_raw);
  const int bh = blockIdx.x, b = bh / p.H, h = bh % p.H;
  const int j = threadIdx.x % D, rg = threadIdx.x / D, r0 = rg * R;
  const int n_ch = (p.T + kChunkF - 1) / kChunkF;
  float C[R];
#pragma unroll
  for (int r = 0; r < R; ++r) C[r] = 0.f;
  Loader<TI, D, NT, kChunkF> ld;
  ld.load(p, b, h, 0);
  ld.store(sm.buf[0]);
  __syncthreads();
  ask_self_chunk<D, NT, kChunkF>(sm.buf[0], p.tau_s);
  TI* Y = reinterpret_cast<TI*>(p.y) + (long long)b * p.sB + (long long)h * p.sH;
  for (int ch = 0; ch < n_ch; ++ch) {
    Chunk<D, kChunkF>& cur = sm.buf[ch & 1];
    const bool more = ch + 1 < n_ch;
    if (more) ld.load(p, b, h, ch + 1);  // in flight while this chunk is computed
    const int nt = min(kChunkF, p.T - ch * kChunkF);
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
      sm.epart[tt][rg][j] = e;
    }
    __syncthreads();  // the chunk's partial reads are complete
    for (int e = threadIdx.x; e < nt * D; e += NT) {  // Answer: Y_t = I~_t + E_t
      const int tt = e / D, jj = e % D;
      float y = cur.vec[tt][3][jj];
#pragma unroll
      for (int g = 0; g < kRG; ++g) y += sm.epart[tt][g][jj];
      stx<TI>(Y + (long long)(ch * kChunkF + tt) * p.sT + jj, y);
    }
    if (more) {
      // nxt held chunk ch - 1, which every thread finished before the barrier above
      Chunk<D, kChunkF>& nxt = sm.buf[(ch + 1) & 1];
      ld.store(nxt);
      __syncthreads();  // also: epart is read above before the next chunk overwrites it
      ask_self_chunk<D, NT, kChunkF>(nxt, p.tau_s);
    }
  }
}

template <typename TI, int D>
cudaError_t fwd_t(const LinearProblem& p, cudaStream_t s) {
  const int smem = (int)sizeof(FwdSmem<D>);
  cudaError_t e = cudaFuncSetAttribute(fwd_kernel<TI, D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) { note_failure("linear forward: shared memory attribute"); return e; }
  fwd_kernel<TI, D><<<(unsigned)(p.B * p.H), kRG * D, smem, s>>>(p);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("linear forward: launch");
  return e;
}

// ---------------------------------------------------------------------------------
// Backward.  Reverse-mode derivative of the recurrent step, in reverse token order, with
// the adjoint dC of the state (S folded into q' = S ^p1 and k' = S ^p2):
//   dI~_t = dY_t + dC_t^T k'_t,   dk'_t = dC_t I~_t,   dq'_t = C^- dY_t,
//   dC^- = dC_t + q'_t dY_t^T,   dalpha_t = rowsum(dC^- * C_{t-1}),   dC_{t-1} = Diag(alpha_t) dC^-
// (C^- = Diag(alpha_t) C_{t-1}); a per-token pass then turns dq', dk' into dp1, dp2
// through the normalisation and S.  kQ threads own row c of the state, a quarter of the
// columns each, so the row sums (dk', dq', dalpha) are two shuffles and the column sum
// (dI~) is reduced across rows by a shuffle reduce-scatter within each warp and shared
// memory across warps.
//   1. checkpoint pass: forward over the tokens, storing the state before every kChunkB
//      tokens in the workspace;
//   2. reverse sweep: tokens staged kStageB at a time; per sub-chunk of kChunkB (last
//      first), the states before each of its tokens are recomputed from the checkpoint into
//      shared memory, then the tokens are walked backwards;
//   3. per-token pass: dp1, dp2.
constexpr int kChunkB = 8;   // tokens per checkpoint / recomputed sub-chunk
constexpr int kStageB = 16;  // tokens per staged chunk (two sub-chunks)
constexpr int kQ = 4;        // threads per state row (each a quarter of the columns)

template <int D>
struct BwdSmem {
  Chunk<D, kStageB> tok;                  // alpha, q', k', I~ of the staged chunk
  float g[kStageB][D];                    // dY of the staged chunk
  float red[kStageB][kQ * D / 32][D];     // per-warp column sums of dC^T k'
  // C_{t-1} of each token of a sub-chunk, each thread's slice as float4s indexed
  // [token][k][thread]: a thread only reads its own slice back, and consecutive lanes
  // touch consecutive 16-byte words (no bank conflicts)
  float4 st[kChunkB][D / (4 * kQ)][kQ * D];
};

template <int D>
__host__ __device__ constexpr long long ckpt_floats(int T) {
  return (long long)((T + kChunkB - 1) / kChunkB) * D * D;
}

template <typename TI, int D>
__global__ void __launch_bounds__(kQ * D) bwd_kernel(LinearProblem p) {
  constexpr int NT = kQ * D, R = D / kQ, NW = NT / 32;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  BwdSmem<D>& sm = *reinterpret_cast<BwdSmem<D>*>(smem_raw);
  const int bh = blockIdx.x, b = bh / p.H, h = bh % p.H;
  const int c = threadIdx.x / kQ, j0 = (threadIdx.x % kQ) * R;
  const bool lead = threadIdx.x % kQ == 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_st = (p.T + kStageB - 1) / kStageB;
  float* ckpt = reinterpret_cast<float*>(p.workspace) + (long long)bh * ckpt_floats<D>(p.T);
  float* dqk = reinterpret_cast<float*>(p.workspace) + (long long)p.B * p.H * ckpt_floats<D>(p.T) +
               (long long)bh * p.T * 2 * D;  // [T][2][D]: dq', dk'
  const long long hb = (long long)b * p.sB + (long long)h * p.sH;
  Loader<TI, D, NT, kStageB> ld;
  auto stage = [&](int sc, bool with_dy) {  // token data of staged chunk sc
    __syncthreads();                         // the previous chunk's data is no longer read
    ld.load(p, b, h, sc);
    ld.store(sm.tok);
    if (with_dy) {
      for (int v4 = threadIdx.x; v4 < kStageB * D / 4; v4 += NT) {
        const int tt = v4 / (D / 4), c4 = (v4 % (D / 4)) * 4, t = sc * kStageB + tt;
        const float4 g = ld4<TI>(reinterpret_cast<const TI*>(p.dy) + hb +
                                 (long long)min(t, p.T - 1) * p.sT + c4);
        *reinterpret_cast<float4*>(&sm.g[tt][c4]) = t < p.T ? g : make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
    __syncthreads();
    ask_self_chunk<D, NT, kStageB>(sm.tok, p.tau_s);
  };
  auto row_step = [&](float (&Cs)[R], int tt) {  // C <- Diag(alpha) C + k' I~^T, own row
    const float a = sm.tok.vec[tt][0][c], kp = sm.tok.vec[tt][2][c];
    const float* I = &sm.tok.vec[tt][3][j0];
#pragma unroll
    for (int i = 0; i < R; i += 4) {
      const float4 i4 = *reinterpret_cast<const float4*>(I + i);
      Cs[i] = fmaf(kp, i4.x, a * Cs[i]);
      Cs[i + 1] = fmaf(kp, i4.y, a * Cs[i + 1]);
      Cs[i + 2] = fmaf(kp, i4.z, a * Cs[i + 2]);
      Cs[i + 3] = fmaf(kp, i4.w, a * Cs[i + 3]);
    }
  };
  // 1. checkpoint pass: the state before every kChunkB tokens
  float C[R];
#pragma unroll
  for (int i = 0; i < R; ++i) C[i] = 0.f;
  for (int sc = 0; sc < n_st; ++sc) {
    const int nt = min(kStageB, p.T - sc * kStageB);
    stage(sc, false);
    for (int tt = 0; tt < nt; ++tt) {
      if (tt % kChunkB == 0) {
        float* ck = ckpt + (long long)((sc * kStageB + tt) / kChunkB) * D * D + c * D + j0;
#pragma unroll
        for (int i = 0; i < R; i += 4)
          *reinterpret_cast<float4*>(ck + i) = make_float4(C[i], C[i + 1], C[i + 2], C[i + 3]);
      }
      row_step(C, tt);
    }
  }
  // 2. reverse sweep
  float dC[R];
#pragma unroll
  for (int i = 0; i < R; ++i) dC[i] = 0.f;
  for (int sc = n_st - 1; sc >= 0; --sc) {
    stage(sc, true);
    const int nt = min(kStageB, p.T - sc * kStageB);
    for (int sub = (nt - 1) / kChunkB; sub >= 0; --sub) {
      const int tb = sub * kChunkB, ns = min(kChunkB, nt - tb);
      const float* ck = ckpt + (long long)((sc * kStageB + tb) / kChunkB) * D * D + c * D + j0;
#pragma unroll
      for (int i = 0; i < R; i += 4) {
        const float4 x = *reinterpret_cast<const float4*>(ck + i);
        C[i] = x.x; C[i + 1] = x.y; C[i + 2] = x.z; C[i + 3] = x.w;
      }
      for (int u = 0; u < ns; ++u) {  // C_{t-1} of each token of the sub-chunk
#pragma unroll
        for (int i = 0; i < R; i += 4)
          sm.st[u][i / 4][threadIdx.x] = make_float4(C[i], C[i + 1], C[i + 2], C[i + 3]);
        if (u + 1 < ns) row_step(C, tb + u);
      }
      for (int u = ns - 1; u >= 0; --u) {
        const int tt = tb + u, t = sc * kStageB + tt;
        const float a = sm.tok.vec[tt][0][c], qp = sm.tok.vec[tt][1][c];
        const float kp = sm.tok.vec[tt][2][c];
        const float* I = &sm.tok.vec[tt][3][j0];
        const float* G = &sm.g[tt][j0];
        float Cp[R];
#pragma unroll
        for (int i = 0; i < R; i += 4) {
          const float4 x = sm.st[u][i / 4][threadIdx.x];
          Cp[i] = x.x; Cp[i + 1] = x.y; Cp[i + 2] = x.z; Cp[i + 3] = x.w;
        }
        float dk = 0.f, dq = 0.f, da = 0.f, col[R];
#pragma unroll
        for (int i = 0; i < R; ++i) {
          const float cp = Cp[i], g = G[i];
          col[i] = dC[i] * kp;              // this row's share of dC^T k'
          dk = fmaf(dC[i], I[i], dk);
          dq = fmaf(a * cp, g, dq);
          const float dcm = fmaf(qp, g, dC[i]);
          da = fmaf(dcm, cp, da);
          dC[i] = a * dcm;                   // dL/dC_{t-1}
        }
#pragma unroll
        for (int o = 1; o < kQ; o <<= 1) {  // the row's kQ threads
          dk += __shfl_xor_sync(0xffffffffu, dk, o);
          dq += __shfl_xor_sync(0xffffffffu, dq, o);
          da += __shfl_xor_sync(0xffffffffu, da, o);
        }
        if (lead) {
          p.dalpha[hb + (long long)t * p.sT + c] = da;
          dqk[(long long)t * 2 * D + c] = dq;
          dqk[(long long)t * 2 * D + D + c] = dk;
        }
        // column sums over the warp's 32 / kQ rows: reduce-scatter over the lane bits above
        // the kQ column threads
        int off = 0, n = R;
#pragma unroll
        for (int m = 16; m >= kQ; m >>= 1) {
          n >>= 1;
          const bool up = (lane & m) != 0;
#pragma unroll
          for (int i = 0; i < R / 2; ++i) {
            if (i < n) {
              const float send = up ? col[i] : col[i + n];
              const float keep = up ? col[i + n] : col[i];
              col[i] = keep + __shfl_xor_sync(0xffffffffu, send, m);
            }
          }
          off += up ? n : 0;
        }
#pragma unroll
        for (int i = 0; i < R / (32 / kQ); ++i) sm.red[tt][warp][j0 + off + i] = col[i];
      }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < nt * D; e += NT) {  // dI~_t = dY_t + dC_t^T k'_t
      const int tt = e / D, jj = e % D, t = sc * kStageB + tt;
      float s2 = sm.g[tt][jj];
#pragma unroll
      for (int w = 0; w < NW; ++w) s2 += sm.red[tt][w][jj];
      stx<TI>(reinterpret_cast<TI*>(p.dv) + hb + (long long)t * p.sT + jj, s2);
    }
  }
}

// dp1, dp2 of every token (one warp per token) from dq', dk' through q' = S p1 / |p1|,
// k' = S p2 / |p2| and S = sigmoid(p1 . p2 / (tau_S sqrt d)).
template <typename TI, int D>
__global__ void __launch_bounds__(256) post_kernel(LinearProblem p) {
  constexpr int PL = D / 32;
  const long long tok = ((long long)blockIdx.x * 256 + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (tok >= (long long)p.B * p.H * p.T) return;
  const int bh = (int)(tok / p.T), t = (int)(tok % p.T), b = bh / p.H, h = bh % p.H;
  const long long off = (long long)b * p.sB + (long long)h * p.sH + (long long)t * p.sT;
  const float* dqk = reinterpret_cast<const float*>(p.workspace) +
                     (long long)p.B * p.H * ckpt_floats<D>(p.T) + ((long long)bh * p.T + t) * 2 * D;
  float x1[PL], x2[PL], g1[PL], g2[PL];
  float s12 = 0.f, s11 = 0.f, s22 = 0.f;
#pragma unroll
  for (int e = 0; e < PL; ++e) {
    const int cc = lane + 32 * e;
    x1[e] = ldx<TI>(reinterpret_cast<const TI*>(p.p1) + off + cc);
    x2[e] = ldx<TI>(reinterpret_cast<const TI*>(p.p2) + off + cc);
    g1[e] = dqk[cc];
    g2[e] = dqk[D + cc];
    s12 = fmaf(x1[e], x2[e], s12);
    s11 = fmaf(x1[e], x1[e], s11);
    s22 = fmaf(x2[e], x2[e], s22);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s12 += __shfl_xor_sync(0xffffffffu, s12, o);
    s11 += __shfl_xor_sync(0xffffffffu, s11, o);
    s22 += __shfl_xor_sync(0xffffffffu, s22, o);
  }
  const float rsd = rsqrtf((float)D);
  const float S = 1.0f / (1.0f + expf(-s12 * rsd / p.tau_s));
  const float in1 = rsqrtf(s11), in2 = rsqrtf(s22);
  // q' = S q^, k' = S k^:  dS = dq' . q^ + dk' . k^,  dq^ = S dq',  dk^ = S dk'
  float a1 = 0.f, a2 = 0.f;  // q^ . dq', k^ . dk'
#pragma unroll
  for (int e = 0; e < PL; ++e) {
    a1 = fmaf(x1[e] * in1, g1[e], a1);
    a2 = fmaf(x2[e] * in2, g2[e], a2);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    a1 += __shfl_xor_sync(0xffffffffu, a1, o);
    a2 += __shfl_xor_sync(0xffffffffu, a2, o);
  }
  const float dS = a1 + a2;
  const float du = dS * S * (1.0f - S) / p.tau_s * rsd;
#pragma unroll
  for (int e = 0; e < PL; ++e) {
    const int cc = lane + 32 * e;
    // d/dp of p / |p| applied to S dq':  S (dq' - q^ (q^ . dq')) / |p|
    const float d1 = S * (g1[e] - x1[e] * in1 * a1) * in1 + du * x2[e];
    const float d2 = S * (g2[e] - x2[e] * in2 * a2) * in2 + du * x1[e];
    stx<TI>(reinterpret_cast<TI*>(p.dp1) + off + cc, d1);
    stx<TI>(reinterpret_cast<TI*>(p.dp2) + off + cc, d2);
  }
}

template <typename TI, int D>
cudaError_t bwd_t(const LinearProblem& p, cudaStream_t s) {
  const int smem = (int)sizeof(BwdSmem<D>);
  cudaError_t e = cudaFuncSetAttribute(bwd_kernel<TI, D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) { note_failure("linear backward: shared memory attribute"); return e; }
  bwd_kernel<TI, D><<<(unsigned)(p.B * p.H), kQ * D, smem, s>>>(p);
  if ((e = cudaGetLastError()) != cudaSuccess) { note_failure("linear backward: launch"); return e; }
  const long long toks = (long long)p.B * p.H * p.T;
  post_kernel<TI, D><<<(unsigned)((toks * 32 + 255) / 256), 256, 0, s>>>(p);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("linear backward: per-token pass");
  return e;
}

}  // namespace lin

size_t linear_bwd_workspace_bytes(int B, int H, int T, int d) {
  const long long per = d == 32 ? lin::ckpt_floats<32>(T) : lin::ckpt_floats<64>(T);
  return (size_t)((long long)B * H * per + (long long)B * H * T * 2 * d) * sizeof(float);
}

cudaError_t launch_linear_bwd(const LinearProblem& p, cudaStream_t s) {
  if (p.dtype == RELATION_F32)
    return p.d == 32 ? lin::bwd_t<float, 32>(p, s) : lin::bwd_t<float, 64>(p, s);
  return p.d == 32 ? lin::bwd_t<__nv_bfloat16, 32>(p, s) : lin::bwd_t<__nv_bfloat16, 64>(p, s);
}

bool linear_supports(relation_dtype dt, int d) {
  return (dt == RELATION_F32 || dt == RELATION_BF16) && (d == 32 || d == 64);
}

cudaError_t launch_linear_fwd(const LinearProblem& p, cudaStream_t s) {
  if (p.dtype == RELATION_F32)
    return p.d == 32 ? lin::fwd_t<float, 32>(p, s) : lin::fwd_t<float, 64>(p, s);
  return p.d == 32 ? lin::fwd_t<__nv_bfloat16, 32>(p, s) : lin::fwd_t<__nv_bfloat16, 64>(p, s);
}

}  // namespace rel
