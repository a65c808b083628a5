// relation_linear_tc.cu -- chunked tensor-core form of the Linear Relation forward
// (Sec. 5.2, Eq. (decayed-relation-state); App. A.4), bf16, d_h 64 or 128.
//
// The recurrence (relation_linear.cu) regrouped into blocks of LT = 128 tokens.  Per head,
// with q'_t = S_t ^p1_t, k'_t = S_t ^p2_t (Ask Self folded into the unit coordinates), the
// channel-wise cumulative log-retention inside a block L_t = sum_{u <= t} log2 alpha_u
// (a_t = 2^{L_t}), and C_0 the state the block starts from (fp32, d x d, kept in TMEM):
//   E_t = (a_t q'_t)^T C_0 + sum_{j < t} (q'_t . (a_t / a_j) k'_j) I~_j,   Y_t = I~_t + E_t
//   C_L = Diag(a_L) C_0 + sum_j ((a_L / a_j) k'_j) I~_j^T
// so that a block is four tcgen05 products:
//   S   = Qm Km^T          Qm_t = q'_t 2^{L_t - L_m}, Km_j = k'_j 2^{L_m - L_j}   (M = N = 128)
//   E   = Qs C_0           Qs_t = q'_t 2^{L_t}
//   E  += tril(S, -1) I~   (S masked and packed to bf16 in TMEM: a TS product)
//   C  <- Diag(2^{L_L}) C + KL^T I~,   KL_j = k'_j 2^{L_L - L_j}
// The ratio a_t / a_j of the intra-block pairs is split at the block's midpoint m (the
// 64th token), so each factor covers at most half a block of decay; the inter-block and
// state factors are at most 1.  A factor beyond 2^120 (a channel decaying below 2^-120
// within 64 tokens) is clamped and the call reports RELATION_ERR_UNSUPPORTED through
// dev_status: the result is then not exact (the recurrent kernels have no such limit).
//
// One CTA per (head, 64 information columns): the columns of C and Y never mix, so a
// d_h = 128 head runs as two CTAs that share the Q / K operands' arithmetic.  Warps 0-3
// (thread = TMEM lane) do Ask Self, the log-retention scans, the operands, the masking,
// the state's decay and bf16 copy, and the output; warp 4 issues the TMA loads, warp 5
// (warp-uniform, elect.sync) the MMAs.  Every mbarrier wait is bounded (common.cuh).
#include <cudaTypedefs.h>
#include <math.h>

#include "relation_linear_tc.cuh"

namespace rel {
namespace lintc {
template <int D>
struct Cfg {
  static constexpr int KB = D / 64;          // 64-channel (128-byte) blocks of a p tile
  static constexpr int PT = LT * D * 2;      // p1 / p2 / operand tile, [128 t][D] bf16
  static constexpr int VT = LT * NC * 2;     // the CTA's 64 columns of I~
  static constexpr int AT = LT * D * 4;      // alpha, [D / 32][128 t][32] fp32
  static constexpr int KLT = LT * 128 * 2;   // KL as a 128-channel tile (d_h = 64: upper half 0)
  static constexpr int C0T = D * NC * 2;     // bf16 copy of C_0's 64 columns, [D c][64 n]
  // Input stages (the next block's loads overlap the current block; one stage at d_h = 128,
  // whose tiles leave no room for a second): p1 (then Qm in place, then the Y staging),
  // p2 (then Km in place), the CTA's I~ columns, alpha (then its running log2 sums).
  static constexpr int STAGES = D == 64 ? 2 : 1;
  static constexpr int OFF_P1 = 0;
  static constexpr int OFF_P2 = OFF_P1 + PT;
  static constexpr int OFF_V = OFF_P2 + PT;
  static constexpr int OFF_A = OFF_V + VT;
  static constexpr int STAGE = 2 * PT + VT + AT;
  static constexpr int OFF_QS = STAGES * STAGE;
  static constexpr int OFF_KL = OFF_QS + PT;
  static constexpr int OFF_C0 = OFF_KL + KLT;  // also the per-token / per-channel scalars
  static constexpr int OFF_BAR = OFF_C0 + C0T;
  static constexpr int SMEM = OFF_BAR + 128 + 1024;
  static constexpr uint32_t LOAD_BYTES = 2 * PT + VT + AT;
};
static_assert(Cfg<64>::SMEM <= 232448 && Cfg<128>::SMEM <= 232448, "shared memory");

template <int D, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    lin_tc_fwd_kernel(const __grid_constant__ CUtensorMap tmP1,
                      const __grid_constant__ CUtensorMap tmP2,
                      const __grid_constant__ CUtensorMap tmV,
                      const __grid_constant__ CUtensorMap tmA,
                      const __grid_constant__ CUtensorMap tmY,
                      const __grid_constant__ CUtensorMap tmC0, LinearProblem p, LinCp cp) {
  using C = Cfg<D>;
  constexpr bool kDelta = MODE == MODE_DELTA || MODE == MODE_BDELTA;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sb = smem_u32(smem);
  auto bar = [&](int i) -> uint32_t { return sb + C::OFF_BAR + 8u * (uint32_t)i; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_BAR + 96);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_BAR + 104);
  int* clamped = reinterpret_cast<int*>(smem + C::OFF_BAR + 108);
  // per-token / per-channel scalars: in the C0 tile's space, or (OUT, where C0 is loaded
  // with the inputs) in KL's, which that mode does not use
  float* sq = reinterpret_cast<float*>(smem + (MODE == MODE_OUT ? C::OFF_KL : C::OFF_C0));
  float* sk = sq + LT;                                             // [128] S_t / |p2_t|
  float* half_sum = sk + LT;                                       // [2][128] (d_h = 64)
  float* lmid_s = half_sum + 2 * LT;                               // [128] L_m per channel
  float* lend_s = lmid_s + LT;                                     // [128] L_end per channel

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int NSPLIT = D / NC;
  const int nb = (p.T + LT - 1) / LT;
  // SEQ: one CTA per (head, split) over blocks [0, nb); DELTA / OUT: one block per CTA
  const int cta_blk = MODE == MODE_SEQ ? 0 : (int)(blockIdx.x % nb);
  const int bhs = MODE == MODE_SEQ ? (int)blockIdx.x : (int)(blockIdx.x / nb);
  const int split = bhs % NSPLIT;
  const int bh = bhs / NSPLIT;
  const int b = bh / p.H, h = bh % p.H;
  const int blk_first = cta_blk, blk_end = MODE == MODE_SEQ ? nb : cta_blk + 1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < NBAR; ++i)  // arrivals of the 128 elementwise threads, or one
      mbar_init(bar(i), (i == B_OPS || i == B_C0 || i == B_A || i == B_EPI || i == B_EPI + 1)
                            ? 128 : 1);
    *abort_flag = 0;
    *clamped = 0;
    fence_mbar_init();
  }
  if (D == 64 && MODE != MODE_OUT) {  // KL's channels 64..127 stay zero (M = 128 product)
    for (int i = threadIdx.x; i < LT * 64 * 2 / 16; i += kThreads)
      *reinterpret_cast<uint4*>(smem + C::OFF_KL + LT * 128 + i * 16) = make_uint4(0, 0, 0, 0);
    fence_async_smem();
  }
  if (warp == 5) tmem_alloc(smem_u32(tmem_slot), kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const Abort ab{abort_flag, p.dev_status};

  if (warp == 4) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmP1);
      tma_prefetch_desc(&tmP2);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmA);
      int issued = 0;
      for (int blk = blk_first; blk < blk_end; ++blk) {
        const int it = blk - blk_first;
        const int st = it % C::STAGES, use = it / C::STAGES;
        // the stage's previous block: its MMAs and its output staging are done
        if (use > 0 && (!mbar_wait(bar(B_FREE + st), (use - 1) & 1, ab) ||
                        !mbar_wait(bar(B_EPI + st), (use - 1) & 1, ab)))
          break;
        const int t0 = blk * LT;
        const uint32_t sg = sb + st * C::STAGE;
        const uint32_t lb = bar(B_LOAD + st);
        mbar_arrive_expect_tx(lb, C::LOAD_BYTES + (MODE == MODE_OUT ? C::C0T : 0));
        if (MODE == MODE_OUT)  // the state the block starts from, in the MN-major B layout
          tma_load_2d(sb + C::OFF_C0, &tmC0, lb, 0, (bhs * (nb + 1) + blk) * D);
        for (int kb = 0; kb < C::KB; ++kb) {
          tma_load_4d(sg + C::OFF_P1 + kb * LT * 128, &tmP1, lb, kb * 64, t0, h, b);
          tma_load_4d(sg + C::OFF_P2 + kb * LT * 128, &tmP2, lb, kb * 64, t0, h, b);
        }
        tma_load_4d(sg + C::OFF_V, &tmV, lb, split * NC, t0, h, b);
        for (int k = 0; k < D / 32; ++k)
          tma_load_4d(sg + C::OFF_A + k * LT * 128, &tmA, lb, k * 32, t0, h, b);
        issued = it + 1;
      }
      if (ab.raised())  // copies in flight land before the CTA releases its shared memory
        for (int it = issued - C::STAGES > 0 ? issued - C::STAGES : 0; it < issued; ++it)
          drain_wait(bar(B_LOAD + it % C::STAGES), (it / C::STAGES) & 1);
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------------ MMA issuer
    constexpr uint32_t id_s = idesc_bf16_f32(128, 128, false, false);
    constexpr uint32_t id_e = idesc_bf16_f32(128, NC, false, true);
    constexpr uint32_t id_c = idesc_bf16_f32(128, NC, true, true);
    bool ok = true;
    for (int blk = blk_first; ok && blk < blk_end; ++blk) {
      const int it = blk - blk_first;
      const uint32_t ph = it & 1;
      const int st = it % C::STAGES;
      const uint32_t sg = sb + st * C::STAGE;
      if (!(ok = mbar_wait_warp(bar(B_OPS), ph, ab))) break;
      tc_fence_after();
      if (!kDelta) {
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {  // S = Qm Km^T
          const uint32_t koff = (kk >> 2) * (LT * 128) + (kk & 3) * 32;
          mma_ss_w(tmem + COL_S, smem_desc_sw128(sg + C::OFF_P1 + koff, 16, 1024),
                   smem_desc_sw128(sg + C::OFF_P2 + koff, 16, 1024), id_s, kk > 0 ? 1u : 0u);
        }
        mma_commit_w(bar(B_S));
        if (!(ok = mbar_wait_warp(bar(B_C0), ph, ab))) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {  // E = Qs C_0
          const uint32_t koff = (kk >> 2) * (LT * 128) + (kk & 3) * 32;
          mma_ss_w(tmem + COL_E, smem_desc_sw128(sb + C::OFF_QS + koff, 16, 1024),
                   smem_desc_sw128(sb + C::OFF_C0 + kk * 16 * 128, D * 128, 1024), id_e,
                   kk > 0 ? 1u : 0u);
        }
        if (!(ok = mbar_wait_warp(bar(B_A), ph, ab))) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < LT / 16; ++kk)  // E += tril(S, -1) I~   (A from TMEM)
          mma_ts_w(tmem + COL_E, tmem + COL_S + kk * 8,
                   smem_desc_sw128(sg + C::OFF_V + kk * 16 * 128, LT * 128, 1024), id_e, 1u);
        mma_commit_w(bar(B_E));
      }
      if (MODE != MODE_OUT) {
        // SEQ: C += KL^T I~ (C decayed by the threads); DELTA: the block's own sum;
        // BDELTA: Qs^T dY
#pragma unroll
        for (int kk = 0; kk < LT / 16; ++kk)
          mma_ss_w(tmem + COL_C, smem_desc_sw128(sb + C::OFF_KL + kk * 16 * 128, LT * 128, 1024),
                   smem_desc_sw128(sg + C::OFF_V + kk * 16 * 128, LT * 128, 1024), id_c,
                   ((MODE == MODE_SEQ && blk > 0) || kk > 0) ? 1u : 0u);
        mma_commit_w(bar(B_STATE));
      }
      mma_commit_w(bar(B_FREE + st));
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ elementwise
    const int t = threadIdx.x;  // token of the block (phases A, D, E) / TMEM lane
    const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
    const float inv_tau_sqrt_d = 1.0f / (p.tau_s * sqrtf((float)D));
    // phase B: thread (c, half) for d_h = 64, thread c over all 128 tokens for d_h = 128
    const int c = D == 64 ? (t & 63) : t;
    const int half = D == 64 ? (t >> 6) : 0;
    constexpr int TPT = D == 64 ? 64 : 128;  // tokens per phase-B thread
    const int tb0 = half * 64;
    uint8_t* p1s = smem + C::OFF_P1;
    uint8_t* p2s = smem + C::OFF_P2;
    float* al = reinterpret_cast<float*>(smem + C::OFF_A);
    auto al_at = [&](int tok, int ch) -> float& {  // [D / 32][128][32] fp32, 128-byte swizzle
      return al[al_swz(tok, ch)];
    };
    float l_end = 0.f;  // this channel's L at the block's last token (phase C, c < D)
    bool ok = true, my_clamp = false;
    for (int blk = blk_first; ok && blk < blk_end; ++blk) {
      const int it = blk - blk_first;
      const uint32_t ph = it & 1;
      const int t0 = blk * LT;
      const int st = it % C::STAGES;
      uint8_t* const sg = smem + st * C::STAGE;
      p1s = sg + C::OFF_P1;
      p2s = sg + C::OFF_P2;
      al = reinterpret_cast<float*>(sg + C::OFF_A);
      ok = __all_sync(0xffffffffu, mbar_wait(bar(B_LOAD + st), (it / C::STAGES) & 1, ab));
      if (!ok) break;
      // ---- phase A: Ask Self of token t (rows past T give zero operands)
      {
        float dot = 0.f, n1 = 0.f, n2 = 0.f;
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb) {
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t off = kb * LT * 128 + t * 128 + ((k ^ (t & 7)) << 4);
            const uint4 a4 = *reinterpret_cast<const uint4*>(p1s + off);
            const uint4 b4 = *reinterpret_cast<const uint4*>(p2s + off);
            const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w}, bw[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&aw[e]));
              const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bw[e]));
              dot = fmaf(x.x, y.x, fmaf(x.y, y.y, dot));
              n1 = fmaf(x.x, x.x, fmaf(x.y, x.y, n1));
              n2 = fmaf(y.x, y.x, fmaf(y.y, y.y, n2));
            }
          }
        }
        float s1 = 0.f, s2 = 0.f;
        if (t0 + t < p.T) {
          const float S = 1.0f / (1.0f + __expf(-dot * inv_tau_sqrt_d));
          s1 = S * rsqrtf(n1);
          s2 = S * rsqrtf(n2);
        }
        sq[t] = s1;
        sk[t] = s2;
      }
      // ---- phase B, pass 1 (thread = channel, d_h = 64: channel and half block): the
      // inclusive running sums L_t of log2 alpha in place of alpha (0 past T)
      // (batches of 16: the loads and logarithms of a batch are issued before its stores)
      float lsum = 0.f, l_mid;
      for (int i0 = 0; i0 < TPT; i0 += 16) {
        float la[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          const int tok = tb0 + i0 + u;
          la[u] = (t0 + tok < p.T) ? __log2f(al_at(tok, c)) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          lsum += la[u];
          al_at(tb0 + i0 + u, c) = lsum;  // d_h = 64, second half: relative to its start
        }
      }
      if (D == 64) half_sum[half * 128 + c] = lsum;
      ew_sync();
      if (D == 64) {
        l_mid = half_sum[c];
        l_end = half_sum[c] + half_sum[128 + c];
      } else {
        l_mid = al_at(63, c);
        l_end = lsum;
      }
      if (t < D) {  // per-channel L_m and L_end for the token-parallel pass
        lmid_s[t] = l_mid;
        lend_s[t] = l_end;
      }
      ew_sync();
      // Qs, KL and the state are single buffers: the last block's state product (the last
      // reader of KL; Qs's reader precedes B_E) must be done before they are written
      if (MODE == MODE_SEQ && blk > 0) {
        ok = __all_sync(0xffffffffu, mbar_wait(bar(B_STATE), (blk - 1) & 1, ab));
        if (!ok) break;
        tc_fence_after();
      }
      // ---- pass 2 (thread = token t, 8 channels per 16-byte access): the four operands,
      // Qm and Km in place of p1 and p2
      {
        const int tok = t;
        const float s1 = sq[tok], s2 = sk[tok];
#pragma unroll
        for (int k = 0; k < D / 8; ++k) {
          const uint32_t off = (k >> 3) * LT * 128 + tok * 128 + (((k & 7) ^ (tok & 7)) << 4);
          const uint4 a4 = *reinterpret_cast<const uint4*>(p1s + off);
          const uint4 b4 = *reinterpret_cast<const uint4*>(p2s + off);
          const float4 L0 = *reinterpret_cast<const float4*>(&al_at(tok, 8 * k));
          const float4 L1 = *reinterpret_cast<const float4*>(&al_at(tok, 8 * k + 4));
          const float4 M0 = *reinterpret_cast<const float4*>(lmid_s + 8 * k);
          const float4 M1 = *reinterpret_cast<const float4*>(lmid_s + 8 * k + 4);
          const float4 E0 = *reinterpret_cast<const float4*>(lend_s + 8 * k);
          const float4 E1 = *reinterpret_cast<const float4*>(lend_s + 8 * k + 4);
          const float Lv[8] = {L0.x, L0.y, L0.z, L0.w, L1.x, L1.y, L1.z, L1.w};
          const float Mv[8] = {M0.x, M0.y, M0.z, M0.w, M1.x, M1.y, M1.z, M1.w};
          const float Ev[8] = {E0.x, E0.y, E0.z, E0.w, E1.x, E1.y, E1.z, E1.w};
          const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w}, bw[4] = {b4.x, b4.y, b4.z, b4.w};
          uint32_t qm[4], km[4], qs[4], kl[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&aw[e]));
            const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bw[e]));
            float r[2][4];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
              const int ch = 2 * e + u;
              // the second half's sums (d_h = 64) are relative to the half's start
              const float L = Lv[ch] + ((D == 64 && tok >= 64) ? Mv[ch] : 0.f);
              float dm = L - Mv[ch];  // log2 of a_t / a_m
              if (fabsf(dm) > kClampLog2) {
                dm = copysignf(kClampLog2, dm);
                my_clamp = true;
              }
              const float xv = u ? x.y : x.x, yv = u ? y.y : y.x;
              if (!kDelta) {
                r[u][0] = xv * s1 * ex2_approx(dm);      // Qm
                r[u][1] = yv * s2 * ex2_approx(-dm);     // Km
                r[u][2] = xv * s1 * ex2_approx(L);       // Qs (factor <= 1)
              }
              if (MODE == MODE_BDELTA)
                r[u][3] = xv * s1 * ex2_approx(L);         // Qs, in KL's place
              else if (MODE != MODE_OUT)
                r[u][3] = yv * s2 * ex2_approx(Ev[ch] - L);  // KL (factor <= 1)
            }
            if (!kDelta) {
              qm[e] = pack_bf16x2(r[0][0], r[1][0]);
              km[e] = pack_bf16x2(r[0][1], r[1][1]);
              qs[e] = pack_bf16x2(r[0][2], r[1][2]);
            }
            if (MODE != MODE_OUT) kl[e] = pack_bf16x2(r[0][3], r[1][3]);
          }
          if (!kDelta) {
            *reinterpret_cast<uint4*>(p1s + off) = make_uint4(qm[0], qm[1], qm[2], qm[3]);
            *reinterpret_cast<uint4*>(p2s + off) = make_uint4(km[0], km[1], km[2], km[3]);
            *reinterpret_cast<uint4*>(smem + C::OFF_QS + off) =
                make_uint4(qs[0], qs[1], qs[2], qs[3]);
          }
          if (MODE != MODE_OUT)
            *reinterpret_cast<uint4*>(smem + C::OFF_KL + off) =
                make_uint4(kl[0], kl[1], kl[2], kl[3]);
        }
      }
      fence_async_smem();
      ew_sync();
      mbar_arrive(bar(B_OPS));
      if (kDelta) {
        // the block's state (adjoint) contribution and decay, to the workspace
        ok = __all_sync(0xffffffffu, mbar_wait(bar(B_STATE), 0, ab));
        if (!ok) break;
        tc_fence_after();
        if (t < D) {
          uint32_t z[64];
          tmem_ld32(trow + COL_C, z);
          tmem_ld32(trow + COL_C + 32, z + 32);
          tmem_ld_wait();
          const long long row = (long long)(bhs * nb + blk) * D + t;
          float4* dst = reinterpret_cast<float4*>(cp.dC + row * 64);
#pragma unroll
          for (int k = 0; k < 16; ++k)
            dst[k] = make_float4(__uint_as_float(z[4 * k]), __uint_as_float(z[4 * k + 1]),
                                 __uint_as_float(z[4 * k + 2]), __uint_as_float(z[4 * k + 3]));
          cp.g[row] = ex2_approx(l_end);
        }
        continue;
      }
      if (MODE == MODE_OUT) {
        mbar_arrive(bar(B_C0));  // C0 came with the block's inputs
      } else {
      // ---- phase C: the state after the last block (complete, waited above), its bf16
      // copy, then decayed by a_L
      if (t < D) {
        uint32_t z[64];
        if (blk > 0) {
          tmem_ld32(trow + COL_C, z);
          tmem_ld32(trow + COL_C + 32, z + 32);
          tmem_ld_wait();
        } else {
#pragma unroll
          for (int n = 0; n < 64; ++n) z[n] = 0u;
        }
        uint8_t* crow = smem + C::OFF_C0 + t * 128;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          uint32_t w[4];
#pragma unroll
          for (int e = 0; e < 4; ++e)
            w[e] = pack_bf16x2(__uint_as_float(z[8 * k + 2 * e]), __uint_as_float(z[8 * k + 2 * e + 1]));
          *reinterpret_cast<uint4*>(crow + ((k ^ (t & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
        }
        if (blk > 0) {
          const float decay = ex2_approx(l_end);
#pragma unroll
          for (int n = 0; n < 64; ++n) z[n] = __float_as_uint(__uint_as_float(z[n]) * decay);
          tmem_st16(trow + COL_C, z);
          tmem_st16(trow + COL_C + 16, z + 16);
          tmem_st16(trow + COL_C + 32, z + 32);
          tmem_st16(trow + COL_C + 48, z + 48);
          tmem_st_wait();
        }
      }
      fence_async_smem();
      tc_fence_before();
      mbar_arrive(bar(B_C0));
      }
      // ---- phase D: S masked to the strictly earlier tokens, packed to bf16 in place
      ok = __all_sync(0xffffffffu, mbar_wait(bar(B_S), ph, ab));
      if (!ok) break;
      tc_fence_after();
#pragma unroll
      for (int c0 = 0; c0 < LT; c0 += 32) {
        uint32_t s[32], pk[16];
        tmem_ld32(trow + COL_S + c0, s);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
          const float lo = (c0 + j < t) ? __uint_as_float(s[j]) : 0.f;
          const float hi = (c0 + j + 1 < t) ? __uint_as_float(s[j + 1]) : 0.f;
          pk[j >> 1] = pack_bf16x2(lo, hi);
        }
        tmem_st16(trow + COL_S + (c0 >> 1), pk);  // columns already read
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(bar(B_A));
      // ---- phase E: Y = I~ + E, staged per warp (32 rows) and stored by TMA
      ok = __all_sync(0xffffffffu, mbar_wait(bar(B_E), ph, ab));
      if (!ok) break;
      tc_fence_after();
      {
        uint32_t z[64];
        tmem_ld32(trow + COL_E, z);
        tmem_ld32(trow + COL_E + 32, z + 32);
        tmem_ld_wait();
        const uint8_t* vrow = sg + C::OFF_V + t * 128;
        uint8_t* ystage = sg + C::OFF_P1 + warp * (32 * 128) + lane * 128;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint4 vv = *reinterpret_cast<const uint4*>(vrow + ((k ^ (t & 7)) << 4));
          const uint32_t vw[4] = {vv.x, vv.y, vv.z, vv.w};
          uint32_t yw[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 vf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&vw[e]));
            yw[e] = pack_bf16x2(vf.x + __uint_as_float(z[8 * k + 2 * e]),
                                vf.y + __uint_as_float(z[8 * k + 2 * e + 1]));
          }
          *reinterpret_cast<uint4*>(ystage + ((k ^ (lane & 7)) << 4)) =
              make_uint4(yw[0], yw[1], yw[2], yw[3]);
        }
        fence_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_4d(&tmY, smem_u32(sg + C::OFF_P1 + warp * (32 * 128)), split * NC,
                       t0 + warp * 32, h, b);
          tma_store_commit();
          tma_store_wait_read_all();  // the staging (the next block's p1) is reloaded next
        }
        __syncwarp();
      }
      mbar_arrive(bar(B_EPI + st));
    }
    if (my_clamp) atomicExch(clamped, 1);
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *clamped && p.dev_status && !*abort_flag)
    atomicExch(p.dev_status, (int)RELATION_ERR_UNSUPPORTED);
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Sequential scan of the state over the blocks of one (head, split), for the chunk-parallel
// forward: C_0(0) = 0, C_0(b + 1) = Diag(g_b) C_0(b) + dC_b, each C_0(b) written in bf16
// (row-major [D][64] per block, the OUT pass's B operand after a swizzled TMA load).  A CTA
// takes 8 channels x 64 columns, two per thread (a warp = one channel's 64 columns,
// coalesced); the loads of the next 8 blocks are in flight while 8 are combined.
//   REV (the backward): from the last block down, the state's adjoint leaving block b,
//   dC(nb - 1) = 0, dC(b - 1) = Diag(g_b) dC(b) + dQ_b (dQ_b = Qs_b^T dY_b in dC's place),
//   written to out_rows (bf16 [nb][D][64] per (head, split)).  Forward: nb + 1 states.
template <int D, bool REV>
__global__ void __launch_bounds__(256) scan_kernel(LinCp cp, __nv_bfloat16* out_rows) {
  constexpr int CPB = 8, P = 8;
  const int cg = (int)(blockIdx.x % (D / CPB));
  const int bhs = (int)(blockIdx.x / (D / CPB));
  const int c = cg * CPB + (int)(threadIdx.x >> 5);
  const int n = (int)(threadIdx.x & 31) * 2;
  const int nb = cp.nb;
  const long long base = (long long)bhs * nb * D + c;  // row of block blk: base + blk D
  // output rows: forward nb + 1 states per (head, split), backward nb adjoints
  const long long obase = (long long)bhs * (REV ? nb : nb + 1) * D + c;
  auto load = [&](int b0, float2 (&dv)[P], float (&gv)[P]) {
#pragma unroll
    for (int u = 0; u < P; ++u) {
      const int blk = REV ? nb - 1 - (b0 + u) : b0 + u;
      if (blk >= 0 && blk < nb) {
        const long long row = base + (long long)blk * D;
        dv[u] = *reinterpret_cast<const float2*>(cp.dC + row * 64 + n);
        gv[u] = cp.g[row];
      } else {
        dv[u] = make_float2(0.f, 0.f);
        gv[u] = 1.f;
      }
    }
  };
  float2 st = make_float2(0.f, 0.f), cur[P];
  float gc[P];
  load(0, cur, gc);
  for (int b0 = 0; b0 < nb; b0 += P) {
    float2 nxt[P];
    float gn[P];
    load(b0 + P, nxt, gn);
#pragma unroll
    for (int u = 0; u < P; ++u) {
      const int i = b0 + u;
      if (i < nb) {
        const int blk = REV ? nb - 1 - i : i;
        const long long orow = obase + (long long)blk * D;
        *reinterpret_cast<__nv_bfloat162*>(out_rows + orow * 64 + n) =
            __floats2bfloat162_rn(st.x, st.y);
        st = make_float2(fmaf(gc[u], st.x, cur[u].x), fmaf(gc[u], st.y, cur[u].y));
      }
    }
#pragma unroll
    for (int u = 0; u < P; ++u) {
      cur[u] = nxt[u];
      gc[u] = gn[u];
    }
  }
  if (!REV)  // the final state, after the last block
    *reinterpret_cast<__nv_bfloat162*>(out_rows + (obase + (long long)nb * D) * 64 + n) =
        __floats2bfloat162_rn(st.x, st.y);
}

// Workspace layout of the chunk-parallel forward: dC and g per (head, split, block), C0 per
// (head, split) and block plus the final state (see LinCp).
static size_t cp_bytes(long long heads, long long nb, int d, LinCp* out, void* base) {
  const long long rows = heads * nb * d, rows_c0 = heads * (nb + 1) * d;
  const size_t b_dc = align256((size_t)rows * 64 * 4), b_g = align256((size_t)rows * 4);
  const size_t b_c0 = align256((size_t)rows_c0 * 64 * 2);
  if (out) {
    uint8_t* q = static_cast<uint8_t*>(base);
    out->dC = reinterpret_cast<float*>(q);
    out->g = reinterpret_cast<float*>(q + b_dc);
    out->c0 = reinterpret_cast<__nv_bfloat16*>(q + b_dc + b_g);
  }
  return b_dc + b_g + b_c0;
}

template <int D>
static cudaError_t fwd_t(const LinearProblem& lp, void* workspace, cudaStream_t s) {
  const int smem = Cfg<D>::SMEM;
  const bool cp_path = workspace != nullptr;
  cudaError_t e;
  for (auto fn : {lin_tc_fwd_kernel<D, MODE_SEQ>, lin_tc_fwd_kernel<D, MODE_DELTA>,
                  lin_tc_fwd_kernel<D, MODE_OUT>})
    if ((e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) !=
        cudaSuccess) {
      note_failure("linear chunked forward: shared memory attribute");
      return e;
    }
  Problem p{};  // the bf16 tensor-map helper's view of the shapes
  p.B = lp.B; p.T = lp.T; p.H = lp.H; p.d = lp.d;
  p.sB = lp.sB; p.sT = lp.sT; p.sH = lp.sH;
  const int nb = (lp.T + LT - 1) / LT;
  const long long heads = (long long)lp.B * lp.H * (D / NC);
  LinCp cp{};
  cp.nb = nb;
  CUtensorMap m1, m2, mv, ma, my, mc;
  if (!tc::make_tmap_bf16(&m1, lp.p1, p, LT) || !tc::make_tmap_bf16(&m2, lp.p2, p, LT) ||
      !tc::make_tmap_bf16(&mv, lp.v, p, LT) || !tc::make_tmap_bf16(&my, lp.y, p, 32) ||
      !make_tmap_alpha(&ma, lp, true)) {
    note_failure("linear chunked forward: TMA descriptors");
    return cudaErrorInvalidValue;
  }
  mc = m1;  // unused by the sequential mode
  if (cp_path) {
    cp_bytes(heads, nb, D, &cp, workspace);
    if (!make_tmap_c0(&mc, cp.c0, heads * (nb + 1) * D, D)) {
      note_failure("linear chunked forward: TMA descriptor of the workspace");
      return cudaErrorInvalidValue;
    }
  }
  if (!cp_path) {
    if (heads > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    lin_tc_fwd_kernel<D, MODE_SEQ><<<(unsigned)heads, kThreads, smem, s>>>(m1, m2, mv, ma, my, mc,
                                                                          lp, cp);
  } else {
    const long long grid = heads * nb;
    if (grid > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    lin_tc_fwd_kernel<D, MODE_DELTA><<<(unsigned)grid, kThreads, smem, s>>>(m1, m2, mv, ma, my, mc,
                                                                           lp, cp);
    if ((e = cudaGetLastError()) != cudaSuccess) { note_failure("linear chunked forward: launch"); return e; }
    scan_kernel<D, false><<<(unsigned)(heads * (D / 8)), 256, 0, s>>>(cp, cp.c0);
    if ((e = cudaGetLastError()) != cudaSuccess) { note_failure("linear chunked forward: launch"); return e; }
    lin_tc_fwd_kernel<D, MODE_OUT><<<(unsigned)grid, kThreads, smem, s>>>(m1, m2, mv, ma, my, mc,
                                                                         lp, cp);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("linear chunked forward: launch");
  return e;
}

// The state passes the chunked backward needs (relation_linear_tc_bwd.cu), in the
// workspace laid out by bwd_bytes: the forward's states entering every block and the final
// one (cp.c0), then the state's adjoint leaving every block (dcb, bf16 [heads][nb][D][64]).
// Four launches: forward DELTA, forward scan, BDELTA (Qs^T dY per block), reverse scan.
size_t bwd_bytes(long long heads, long long nb, int d, LinCp* cp, __nv_bfloat16** dcb,
                 void* base) {
  const size_t f = cp_bytes(heads, nb, d, cp, base);
  if (dcb) *dcb = reinterpret_cast<__nv_bfloat16*>(static_cast<uint8_t*>(base) + f);
  return f + align256((size_t)(heads * nb * d) * 64 * 2);
}

template <int D>
cudaError_t states_t(const LinearProblem& lp, const void* dy, void* workspace, cudaStream_t s) {
  const int smem = Cfg<D>::SMEM;
  cudaError_t e;
  for (auto fn : {lin_tc_fwd_kernel<D, MODE_DELTA>, lin_tc_fwd_kernel<D, MODE_BDELTA>})
    if ((e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) !=
        cudaSuccess) {
      note_failure("linear chunked backward: shared memory attribute");
      return e;
    }
  Problem p{};
  p.B = lp.B; p.T = lp.T; p.H = lp.H; p.d = lp.d;
  p.sB = lp.sB; p.sT = lp.sT; p.sH = lp.sH;
  const int nb = (lp.T + LT - 1) / LT;
  const long long heads = (long long)lp.B * lp.H * (D / NC);
  LinCp cp{};
  cp.nb = nb;
  __nv_bfloat16* dcb = nullptr;
  bwd_bytes(heads, nb, D, &cp, &dcb, workspace);
  CUtensorMap m1, m2, mv, mg, ma;
  if (!tc::make_tmap_bf16(&m1, lp.p1, p, LT) || !tc::make_tmap_bf16(&m2, lp.p2, p, LT) ||
      !tc::make_tmap_bf16(&mv, lp.v, p, LT) || !tc::make_tmap_bf16(&mg, dy, p, LT) ||
      !make_tmap_alpha(&ma, lp, true)) {
    note_failure("linear chunked backward: TMA descriptors");
    return cudaErrorInvalidValue;
  }
  const long long grid = heads * nb;
  if (grid > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  // (the Y map is unused in these modes; m1 stands in)
  lin_tc_fwd_kernel<D, MODE_DELTA><<<(unsigned)grid, kThreads, smem, s>>>(m1, m2, mv, ma, m1, m1,
                                                                         lp, cp);
  if ((e = cudaGetLastError()) != cudaSuccess) { note_failure("linear chunked backward: launch"); return e; }
  scan_kernel<D, false><<<(unsigned)(heads * (D / 8)), 256, 0, s>>>(cp, cp.c0);
  if ((e = cudaGetLastError()) != cudaSuccess) { note_failure("linear chunked backward: launch"); return e; }
  lin_tc_fwd_kernel<D, MODE_BDELTA><<<(unsigned)grid, kThreads, smem, s>>>(m1, m2, mg, ma, m1, m1,
                                                                          lp, cp);
  if ((e = cudaGetLastError()) != cudaSuccess) { note_failure("linear chunked backward: launch"); return e; }
  scan_kernel<D, true><<<(unsigned)(heads * (D / 8)), 256, 0, s>>>(cp, dcb);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("linear chunked backward: launch");
  return e;
}
template cudaError_t states_t<64>(const LinearProblem&, const void*, void*, cudaStream_t);

}  // namespace lintc

bool linear_tc_supports(const LinearProblem& p) {
  return p.dtype == RELATION_BF16 && (p.d == 64 || p.d == 128) && p.sB % 8 == 0 &&
         p.sT % 8 == 0 && p.sH % 8 == 0;
}

size_t linear_tc_workspace_bytes(const LinearProblem& p) {
  if (!linear_tc_supports(p)) return 0;
  const long long heads = (long long)p.B * p.H * (p.d / lintc::NC);
  const long long nb = (p.T + lintc::LT - 1) / lintc::LT;
  return lintc::cp_bytes(heads, nb, p.d, nullptr, nullptr);
}

cudaError_t launch_linear_tc_fwd(const LinearProblem& p, void* workspace, cudaStream_t s) {
  if (!linear_tc_supports(p)) return cudaErrorInvalidValue;
  return p.d == 64 ? lintc::fwd_t<64>(p, workspace, s) : lintc::fwd_t<128>(p, workspace, s);
}

}  // namespace rel
