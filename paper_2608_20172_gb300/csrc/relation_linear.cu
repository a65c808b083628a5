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
// kernels therefore split a head's columns across several CTAs (no exchange between them;
// each runs Ask Self for the whole token).  In the forward a column belongs to RG threads,
// each keeping R = d / RG of its rows in registers; a token costs 3 R multiply-adds per
// thread (the read is summed over the column's threads once per chunk).  A CTA walks the
// tokens in order; tokens are staged through shared memory in double-buffered chunks, Ask
// Self (S_t, 1/|p1_t|, 1/|p2_t|) being taken on the way in, by shuffles among the threads
// that load a token, and folded into the coordinates (q'_t = S_t ^p1_t, k'_t = S_t ^p2_t).
// Loads are 4-element vectors without conditions.
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
  float vec[NTOK][4][D];  // [0] alpha, [1] q' = S ^p1, [2] k' = S ^p2, [3] I~
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
  // Ask Self on the way to shared memory: the D / 4 consecutive threads holding a token's
  // vectors reduce p1 . p2, |p1|^2, |p2|^2 by shuffles, and each scales its pieces into
  // q' = S_t p1 / |p1|, k' = S_t p2 / |p2| with S_t = sigmoid(p1 . p2 / (tau_S sqrt d)).
  __device__ __forceinline__ void store(Chunk<D, NTOK>& s, float tau_s) const {
    const float inv_t = 1.0f / (tau_s * sqrtf((float)D));
#pragma unroll
    for (int n = 0; n < NV; ++n) {
      const int v = n * NT + (int)threadIdx.x;
      const int tt = v / (D / 4), c4 = (v % (D / 4)) * 4;
      const float4 a = r[1][n], k = r[2][n];
      float s12 = a.x * k.x + a.y * k.y + a.z * k.z + a.w * k.w;
      float s11 = a.x * a.x + a.y * a.y + a.z * a.z + a.w * a.w;
      float s22 = k.x * k.x + k.y * k.y + k.z * k.z + k.w * k.w;
#pragma unroll
      for (int o = 1; o < D / 4; o <<= 1) {
        s12 += __shfl_xor_sync(0xffffffffu, s12, o);
        s11 += __shfl_xor_sync(0xffffffffu, s11, o);
        s22 += __shfl_xor_sync(0xffffffffu, s22, o);
      }
      const float S = 1.0f / (1.0f + expf(-s12 * inv_t));
      const float f1 = s11 > 0.f ? S * rsqrtf(s11) : 0.f;
      const float f2 = s22 > 0.f ? S * rsqrtf(s22) : 0.f;
      *reinterpret_cast<float4*>(&s.vec[tt][0][c4]) = r[0][n];
      *reinterpret_cast<float4*>(&s.vec[tt][1][c4]) = make_float4(a.x * f1, a.y * f1, a.z * f1, a.w * f1);
      *reinterpret_cast<float4*>(&s.vec[tt][2][c4]) = make_float4(k.x * f2, k.y * f2, k.z * f2, k.w * f2);
      *reinterpret_cast<float4*>(&s.vec[tt][3][c4]) = r[3][n];
    }
  }
};

// Forward: NS CTAs per head, each owning NC = D / NS information columns (the columns
// evolve independently, so the split needs no exchange; every CTA runs Ask Self for the
// whole token).  RG threads per column: thread (j, rg) = tid % NC, tid / NC keeps rows
// rg * R .. + R of column j in registers.  Threads of a warp share at most two row groups,
// so the per-token alpha, q', k' reads are shared-memory broadcasts, and each thread's
// partial read goes to shared memory: Y_t = I~_t + sum_rg e_rg is formed per chunk (the
// output does not feed back into the recurrence), with no per-token shuffle.
constexpr int kChunkF = 16;  // tokens per staged chunk (forward)

template <int D, int NS>
struct FwdCfg {
  static constexpr int NT = D == 32 ? 128 : 256;  // threads
  static constexpr int NC = D / NS;               // columns per CTA
  static constexpr int RG = NT / NC;              // row groups
  static constexpr int R = D / RG;                // rows per thread
  static_assert(R % 4 == 0 && RG * R == D, "row split");
};

template <int D, int NS>
struct FwdSmem {
  Chunk<D, kChunkF> buf[2];
  float epart[kChunkF][FwdCfg<D, NS>::RG][FwdCfg<D, NS>::NC];  // partial reads
};

template <typename TI, int D, int NS>
__global__ void __launch_bounds__(FwdCfg<D, NS>::NT) fwd_kernel(LinearProblem p) {
  using F = FwdCfg<D, NS>;
  constexpr int NT = F::NT, NC = F::NC, RG = F::RG, R = F::R;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  FwdSmem<D, NS>& sm = *reinterpret_cast<FwdSmem<D, NS>*>(smem_raw);
  const int bh = blockIdx.x / NS, js = blockIdx.x % NS, b = bh / p.H, h = bh % p.H;
  const int jl = threadIdx.x % NC, rg = threadIdx.x / NC, r0 = rg * R;
  const int j = js * NC + jl;  // this thread's column of C
  const int n_ch = (p.T + kChunkF - 1) / kChunkF;
  float C[R];
#pragma unroll
  for (int r = 0; r < R; ++r) C[r] = 0.f;
  // Chunk c is loaded into registers two chunks ahead, by loader c % 2, while chunk c - 2
  // is computed, and stored to shared memory once chunk c - 1 is done.
  Loader<TI, D, NT, kChunkF> ld0, ld1;
  ld0.load(p, b, h, 0);
  if (n_ch > 1) ld1.load(p, b, h, 1);
  ld0.store(sm.buf[0], p.tau_s);
  __syncthreads();
  TI* Y = reinterpret_cast<TI*>(p.y) + (long long)b * p.sB + (long long)h * p.sH;
  // chunk ch; `nxt` holds chunk ch + 1, `fre` takes chunk ch + 2
  auto chunk = [&](int ch, Loader<TI, D, NT, kChunkF>& nxt, Loader<TI, D, NT, kChunkF>& fre) {
    Chunk<D, kChunkF>& cur = sm.buf[ch & 1];
    if (ch + 2 < n_ch) fre.load(p, b, h, ch + 2);  // in flight for two chunks
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
      sm.epart[tt][rg][jl] = e;
    }
    __syncthreads();  // the chunk's partial reads are complete
    for (int e = threadIdx.x; e < nt * NC; e += NT) {  // Answer: Y_t = I~_t + E_t
      const int tt = e / NC, cl = e % NC;
      float y = cur.vec[tt][3][js * NC + cl];
#pragma unroll
      for (int g = 0; g < RG; ++g) y += sm.epart[tt][g][cl];
      stx<TI>(Y + (long long)(ch * kChunkF + tt) * p.sT + js * NC + cl, y);
    }
    if (ch + 1 < n_ch) {
      // buffer (ch + 1) & 1 held chunk ch - 1, which every thread finished before the
      // barrier above
      nxt.store(sm.buf[(ch + 1) & 1], p.tau_s);
      __syncthreads();  // also: epart is read above before the next chunk overwrites it
    }
  };
  for (int ch = 0; ch < n_ch; ch += 2) {
    chunk(ch, ld1, ld0);
    if (ch + 1 < n_ch) chunk(ch + 1, ld0, ld1);
  }
}

// column splits of the forward: 16 columns per CTA (d_h = 32: 2 CTAs per head, 64: 4,
// 128: 8)
template <int D>
constexpr int fwd_splits() { return D / 16; }

template <typename TI, int D>
cudaError_t fwd_t(const LinearProblem& p, cudaStream_t s) {
  constexpr int NS = fwd_splits<D>();
  const int smem = (int)sizeof(FwdSmem<D, NS>);
  cudaError_t e = cudaFuncSetAttribute(fwd_kernel<TI, D, NS>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) { note_failure("linear forward: shared memory attribute"); return e; }
  fwd_kernel<TI, D, NS><<<(unsigned)(p.B * p.H * NS), FwdCfg<D, NS>::NT, smem, s>>>(p);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("linear forward: launch");
  return e;
}

// ---------------------------------------------------------------------------------
// Backward.  Reverse-mode derivative of the recurrent step, in reverse token order, with
// the adjoint dC of the state (S folded into q' = S ^p1 and k' = S ^p2):
//   dI~_t = dY_t + dC_t^T k'_t,   dk'_t = dC_t I~_t,   dq'_t = C^- dY_t,
//   dC^- = dC_t + q'_t dY_t^T,   dalpha_t = rowsum(dC^- * C_{t-1}),   dC_{t-1} = Diag(alpha_t) dC^-
// (C^- = Diag(alpha_t) C_{t-1}); a per-token pass then turns dq', dk' into dp1, dp2
// through the normalisation and S.  NS CTAs per head each own NC = D / NS columns of the
// state (and of dC): the column sum (dI~) stays within a CTA, the row sums (dk', dq',
// dalpha) are partial sums over the CTA's columns, added up by the per-token pass.  kQ
// threads own row c of the CTA's columns, a quarter each, so a row sum is two shuffles
// and the column sum is reduced across rows by a shuffle reduce-scatter within each warp
// and shared memory across warps.
//   1. checkpoint pass: forward over the tokens, storing the state before every kChunkB
//      tokens in the workspace;
//   2. reverse sweep: tokens staged kStageB at a time; per sub-chunk of kChunkB (last
//      first), the states before each of its tokens are recomputed from the checkpoint into
//      shared memory, then the tokens are walked backwards;
//   3. per-token pass: dalpha and, through the normalisation and S, dp1, dp2.
constexpr int kChunkB = 8;   // tokens per checkpoint / recomputed sub-chunk
constexpr int kStageB = 16;  // tokens per staged chunk (two sub-chunks)
constexpr int kQ = 4;        // threads per state row (each a quarter of the columns)

// column splits of the backward: 32 columns per CTA (d_h = 32: one CTA per head, 64: 2,
// 128: 4; the reduce-scatter below needs R = NC / kQ >= 32 / kQ)
template <int D>
constexpr int bwd_splits() { return D / 32; }

template <int D>
struct BwdSmem {
  static constexpr int NC = D / bwd_splits<D>();
  Chunk<D, kStageB> tok;                  // alpha, q', k', I~ of the staged chunk
  float g[kStageB][D];                    // dY of the staged chunk
  float red[kStageB][kQ * D / 32][NC];    // per-warp column sums of dC^T k'
  // C_{t-1} of each token of a sub-chunk, each thread's slice as float4s indexed
  // [token][k][thread]: a thread only reads its own slice back, and consecutive lanes
  // touch consecutive 16-byte words (no bank conflicts)
  float4 st[kChunkB][NC / (4 * kQ)][kQ * D];
};

// checkpointed state of one head (all column splits together)
template <int D>
__host__ __device__ constexpr long long ckpt_floats(int T) {
  return (long long)((T + kChunkB - 1) / kChunkB) * D * D;
}

template <typename TI, int D>
__global__ void __launch_bounds__(kQ * D) bwd_kernel(LinearProblem p) {
  constexpr int NS = bwd_splits<D>(), NC = D / NS;
  constexpr int NT = kQ * D, R = NC / kQ, NW = NT / 32;
  static_assert(R >= 32 / kQ && R % 4 == 0, "reduce-scatter over the warp's rows");
  extern __shared__ __align__(16) uint8_t smem_raw[];
  BwdSmem<D>& sm = *reinterpret_cast<BwdSmem<D>*>(smem_raw);
  const int bh = blockIdx.x / NS, js = blockIdx.x % NS, b = bh / p.H, h = bh % p.H;
  const int c = threadIdx.x / kQ, jl0 = (threadIdx.x % kQ) * R;  // row; first local column
  const int j0 = js * NC + jl0;                                  // first column of C
  const bool lead = threadIdx.x % kQ == 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_st = (p.T + kStageB - 1) / kStageB;
  // checkpoints of this CTA's columns: [n_ck][D rows][NC]
  float* ckpt = reinterpret_cast<float*>(p.workspace) + (long long)bh * ckpt_floats<D>(p.T) +
                (long long)js * (ckpt_floats<D>(p.T) / NS);
  // partial row sums over this CTA's columns, [T][3][D]: dq', dk', dalpha
  float* dqk = reinterpret_cast<float*>(p.workspace) + (long long)p.B * p.H * ckpt_floats<D>(p.T) +
               ((long long)bh * NS + js) * p.T * 3 * D;
  const long long hb = (long long)b * p.sB + (long long)h * p.sH;
  // The token data of the next staged chunk is loaded into registers (fetch) while the
  // current one is processed, and stored to shared memory when it is due (stage).
  static_assert(kStageB * D / 4 == NT, "one dY vector per thread and chunk");
  Loader<TI, D, NT, kStageB> ld;
  float4 gpre = make_float4(0.f, 0.f, 0.f, 0.f);  // this thread's dY vector
  auto fetch = [&](int sc, bool with_dy) {
    ld.load(p, b, h, sc);
    if (with_dy) {
      const int tt = threadIdx.x / (D / 4), c4 = (threadIdx.x % (D / 4)) * 4, t = sc * kStageB + tt;
      const float4 g = ld4<TI>(reinterpret_cast<const TI*>(p.dy) + hb +
                               (long long)min(t, p.T - 1) * p.sT + c4);
      gpre = t < p.T ? g : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  };
  auto stage = [&](bool with_dy) {  // the fetched chunk into shared memory
    __syncthreads();                 // the previous chunk's data is no longer read
    ld.store(sm.tok, p.tau_s);
    if (with_dy)
      *reinterpret_cast<float4*>(&sm.g[threadIdx.x / (D / 4)][(threadIdx.x % (D / 4)) * 4]) = gpre;
    __syncthreads();
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
  fetch(0, false);
  for (int sc = 0; sc < n_st; ++sc) {
    const int nt = min(kStageB, p.T - sc * kStageB);
    stage(false);
    if (sc + 1 < n_st) fetch(sc + 1, false);
    else fetch(n_st - 1, true);  // the reverse sweep's first chunk
    for (int tt = 0; tt < nt; ++tt) {
      if (tt % kChunkB == 0) {
        float* ck = ckpt + (long long)((sc * kStageB + tt) / kChunkB) * D * NC + c * NC + jl0;
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
    stage(true);
    if (sc > 0) fetch(sc - 1, true);
    const int nt = min(kStageB, p.T - sc * kStageB);
    for (int sub = (nt - 1) / kChunkB; sub >= 0; --sub) {
      const int tb = sub * kChunkB, ns = min(kChunkB, nt - tb);
      const float* ck = ckpt + (long long)((sc * kStageB + tb) / kChunkB) * D * NC + c * NC + jl0;
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
          dqk[(long long)t * 3 * D + c] = dq;
          dqk[(long long)t * 3 * D + D + c] = dk;
          dqk[(long long)t * 3 * D + 2 * D + c] = da;
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
        for (int i = 0; i < R / (32 / kQ); ++i) sm.red[tt][warp][jl0 + off + i] = col[i];
      }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < nt * NC; e += NT) {  // dI~_t = dY_t + dC_t^T k'_t
      const int tt = e / NC, cl = e % NC, t = sc * kStageB + tt;
      float s2 = sm.g[tt][js * NC + cl];
#pragma unroll
      for (int w = 0; w < NW; ++w) s2 += sm.red[tt][w][cl];
      stx<TI>(reinterpret_cast<TI*>(p.dv) + hb + (long long)t * p.sT + js * NC + cl, s2);
    }
  }
}

// dalpha, dp1, dp2 of every token (one warp per token): the column splits' partial sums of
// dalpha, dq', dk' added up, then dq', dk' taken through q' = S p1 / |p1|,
// k' = S p2 / |p2| and S = sigmoid(p1 . p2 / (tau_S sqrt d)).
template <typename TI, int D>
__global__ void __launch_bounds__(256) post_kernel(LinearProblem p) {
  constexpr int PL = D / 32;
  const long long tok = ((long long)blockIdx.x * 256 + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (tok >= (long long)p.B * p.H * p.T) return;
  const int bh = (int)(tok / p.T), t = (int)(tok % p.T), b = bh / p.H, h = bh % p.H;
  const long long off = (long long)b * p.sB + (long long)h * p.sH + (long long)t * p.sT;
  constexpr int NS = bwd_splits<D>();
  const float* dqk = reinterpret_cast<const float*>(p.workspace) +
                     (long long)p.B * p.H * ckpt_floats<D>(p.T) + ((long long)bh * NS * p.T + t) * 3 * D;
  float x1[PL], x2[PL], g1[PL], g2[PL];
  float s12 = 0.f, s11 = 0.f, s22 = 0.f;
#pragma unroll
  for (int e = 0; e < PL; ++e) {
    const int cc = lane + 32 * e;
    x1[e] = ldx<TI>(reinterpret_cast<const TI*>(p.p1) + off + cc);
    x2[e] = ldx<TI>(reinterpret_cast<const TI*>(p.p2) + off + cc);
    g1[e] = 0.f;
    g2[e] = 0.f;
    float da = 0.f;
#pragma unroll
    for (int js = 0; js < NS; ++js) {
      const float* part = dqk + (long long)js * p.T * 3 * D;
      g1[e] += part[cc];
      g2[e] += part[D + cc];
      da += part[2 * D + cc];
    }
    p.dalpha[off + cc] = da;
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
  bwd_kernel<TI, D><<<(unsigned)(p.B * p.H * bwd_splits<D>()), kQ * D, smem, s>>>(p);
  if ((e = cudaGetLastError()) != cudaSuccess) { note_failure("linear backward: launch"); return e; }
  const long long toks = (long long)p.B * p.H * p.T;
  post_kernel<TI, D><<<(unsigned)((toks * 32 + 255) / 256), 256, 0, s>>>(p);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("linear backward: per-token pass");
  return e;
}

}  // namespace lin

size_t linear_bwd_workspace_bytes(int B, int H, int T, int d) {
  const long long per = (long long)((T + lin::kChunkB - 1) / lin::kChunkB) * d * d;
  const int ns = d / 32;  // bwd_splits
  return (size_t)((long long)B * H * per + (long long)B * H * ns * T * 3 * d) * sizeof(float);
}

cudaError_t launch_linear_bwd(const LinearProblem& p, cudaStream_t s) {
  if (p.dtype == RELATION_F32)
    return p.d == 32 ? lin::bwd_t<float, 32>(p, s)
                     : p.d == 64 ? lin::bwd_t<float, 64>(p, s) : lin::bwd_t<float, 128>(p, s);
  return p.d == 32 ? lin::bwd_t<__nv_bfloat16, 32>(p, s)
                   : p.d == 64 ? lin::bwd_t<__nv_bfloat16, 64>(p, s)
                               : lin::bwd_t<__nv_bfloat16, 128>(p, s);
}

bool linear_supports(relation_dtype dt, int d) {
  return (dt == RELATION_F32 || dt == RELATION_BF16) && (d == 32 || d == 64 || d == 128);
}

cudaError_t launch_linear_fwd(const LinearProblem& p, cudaStream_t s) {
  if (p.dtype == RELATION_F32)
    return p.d == 32 ? lin::fwd_t<float, 32>(p, s)
                     : p.d == 64 ? lin::fwd_t<float, 64>(p, s) : lin::fwd_t<float, 128>(p, s);
  return p.d == 32 ? lin::fwd_t<__nv_bfloat16, 32>(p, s)
                   : p.d == 64 ? lin::fwd_t<__nv_bfloat16, 64>(p, s)
                               : lin::fwd_t<__nv_bfloat16, 128>(p, s);
}

}  // namespace rel
