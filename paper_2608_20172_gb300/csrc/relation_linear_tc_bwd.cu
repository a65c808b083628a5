// relation_linear_tc_bwd.cu -- chunked tensor-core backward of Linear Relation (Sec. 5.2,
// App. A.4; the paper writes out the forward only), bf16, d_h = 64.
//
// Reverse mode through the 128-token blocks of relation_linear_tc.cu, every block in
// parallel.  The state passes come first (relation_linear_tc.cu, states_t): the state C_0
// entering every block and the final one (forward DELTA + scan), and the state's adjoint
// dC leaving every block, dC(b - 1) = Diag(a_L(b)) dC(b) + Qs_b^T dY_b (BDELTA + reverse
// scan).  Then one CTA per block, with G = dY, A = tril(Qm Km^T, -1), dA = tril(G I~^T, -1):
//   X  = dA Km + G (2^{L_m} C_0)^T        dq'_t = 2^{L_t - L_m} X_t
//   Y  = dA^T Qm + Ys,  Ys = I~ (2^{L_end - L_m} dC)^T   dk'_j = 2^{L_m - L_j} Y_j
//   dI~ = G + A^T G + KL dC
//   dL_t = q'_t * dq'_t - k'_t * dk'_t = Qm_t * X_t - Km_t * Y_t
//          (+ sum_n dC[c][n] C_L[c][n] at the block's end, C_L = 2^{L_end} C_0 + KL^T I~,
//           taken as sum_n (2^{L_m} C_0)[c][n] (2^{L_end - L_m} dC)[c][n] + sum_j Km_j * Ys_j)
//   dalpha_u = (sum_{t >= u} dL_t) / alpha_u           (L_t = sum_{u <= t} log2 alpha_u)
// (the midpoint L_m cancels in every product S_tj, so it carries no gradient), and dp1,
// dp2 from dq', dk' through S_t and the normalisation of p1, p2.
// The suffix sums of dL cancel: every pair (t, j) with both tokens at or after u enters
// once through Qm_t X_t and once, negated, through Km_j Y_j, and every Km_j Ys_j once in the
// end term; only the pairs that straddle u survive, and those carry the factor alpha_u that
// the division takes out.  So dL is formed from the very bf16 values of Qm and Km that the
// products read (recomputed bit for bit), and the end term from the same Ys: the pairs
// then cancel up to fp32 rounding, where rounding Qm and Km independently of q' and k'
// would leave errors of the bf16 unit, divided by alpha_u.  The products are tcgen05
// MMAs with fp32 accumulation in TMEM; the masked A and dA go through shared memory so that
// the transposed products read them as MN-major operands.  Warps 0-3 (thread = token or
// channel) do the elementwise work, warp 4 the TMA loads and stores, warp 5 (warp-uniform,
// elect.sync) the MMAs.  Every mbarrier wait is bounded (common.cuh).
#include "relation_linear_tc.cuh"

namespace rel {
namespace lintc {
namespace bwd {

constexpr int D = 64;
constexpr int kTmemCols = 512;  // scratch S / dA 128 | X 64 | Y 64 | dI~ 64 | Ys 64
constexpr int COL_SC = 0, COL_X = 128, COL_Y = 192, COL_DI = 256, COL_YS = 320;
// shared memory (bytes): 128-token tiles of 64 bf16 columns are 16 KB
constexpr int T16 = LT * 64 * 2;
constexpr int OFF_P1 = 0;                 // p1, then Qm in place, then p1 again, then dp1
constexpr int OFF_P2 = OFF_P1 + T16;      // p2, then Km in place, then p2 again, then dp2
constexpr int OFF_V = OFF_P2 + T16;       // I~
constexpr int OFF_G = OFF_V + T16;        // dY, then dI~ (the dv output)
constexpr int OFF_AL = OFF_G + T16;       // alpha, then its running log2 sums [2][128][32] fp32
constexpr int OFF_KL = OFF_AL + LT * 64 * 4;  // KL; from the epilogue on, dL and Km Ys [t][GS]
constexpr int OFF_AS = OFF_KL + T16;      // A = tril(S) [t][j] (2 blocks), then dL [t][64] fp32
constexpr int OFF_DAS = OFF_AS + 2 * T16; // dA [t][j]
constexpr int C64 = 64 * 64 * 2;          // a [64 c][64 n] bf16 tile
constexpr int OFF_C0 = OFF_DAS + 2 * T16; // C_0, then 2^{L_m} C_0 in place
constexpr int OFF_DC = OFF_C0 + C64;      // dC (the state's adjoint leaving the block)
constexpr int OFF_DCP = OFF_DC + C64;     // 2^{L_end - L_m} dC
constexpr int OFF_SC = OFF_DCP + C64;     // scalars, 9 x 128 fp32
constexpr int OFF_BAR = OFF_SC + 9 * LT * 4;
constexpr int SMEM = OFF_BAR + 128 + 1024;
static_assert(SMEM <= 232448, "shared memory");
constexpr uint32_t LOAD_BYTES = 4 * T16 + LT * 64 * 4 + 2 * C64;
constexpr int GS = 68;  // row stride (floats) of the epilogue's [t][64] arrays: float4 rows
constexpr int OFF_GL = OFF_KL, OFF_TS = OFF_GL + LT * GS * 4;
static_assert(OFF_TS + LT * GS * 4 <= OFF_C0, "epilogue arrays overlap the state tiles");

// Qm and Km of one channel as the products read them (bf16), from p1, p2 (bf16 values),
// S / |p|, and the channel's log2 ratio to the midpoint; the epilogue recomputes them
// through this same function, bit for bit.
__device__ __forceinline__ float dm_of(float lv, float lm, bool later, bool& clamped) {
  // log2 of a_t / a_m for one channel from its stored running sum (relative to the block's
  // start, or in the later half to the midpoint) and L_m, clamped to +-kClampLog2
  float dm = (lv + (later ? lm : 0.f)) - lm;
  if (fabsf(dm) > kClampLog2) {
    dm = copysignf(kClampLog2, dm);
    clamped = true;
  }
  return dm;
}
__device__ __forceinline__ void qm_km(float x, float y, float s1, float s2, float dm, float& qm,
                                      float& km) {
  qm = __bfloat162float(__float2bfloat16_rn(x * s1 * ex2_approx(dm)));
  km = __bfloat162float(__float2bfloat16_rn(y * s2 * ex2_approx(-dm)));
}

// Retention below this takes dalpha from the state and its adjoint at the token (phase F).
constexpr float kSmallAlpha = 1.0f / 1024.0f;

// The small-retention fix-up's tiles (dY, p1, p2 loaded again), over the epilogue's dL and
// Km Ys arrays once phase F has read them
constexpr int OFF_FIX_G = OFF_KL, OFF_FIX_P1 = OFF_KL + T16, OFF_FIX_P2 = OFF_KL + 2 * T16;
static_assert(OFF_FIX_P2 + T16 <= OFF_C0 && OFF_KL % 1024 == 0, "fix-up tiles");

enum : int { B_LOAD = 0, B_OPS, B_S, B_A, B_DA, B_DAS, B_MM, B_RELOAD, B_FIX, NBAR };

// Some lane of the warp has a token flagged in its 64-bit mask.
__device__ __forceinline__ bool small_any_warp(unsigned long long m) {
  return __any_sync(0xffffffffu, m != 0ull);
}

__global__ void __launch_bounds__(kThreads, 1)
    lin_tc_bwd_kernel(const __grid_constant__ CUtensorMap tmP1,
                      const __grid_constant__ CUtensorMap tmP2,
                      const __grid_constant__ CUtensorMap tmV,
                      const __grid_constant__ CUtensorMap tmG,
                      const __grid_constant__ CUtensorMap tmA,
                      const __grid_constant__ CUtensorMap tmC0,  // states: [heads][nb + 1][64][64]
                      const __grid_constant__ CUtensorMap tmDC,  // adjoints: [heads][nb][64][64]
                      const __grid_constant__ CUtensorMap tmDP1,
                      const __grid_constant__ CUtensorMap tmDP2,
                      const __grid_constant__ CUtensorMap tmDV, LinearProblem p, int nb) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sb = smem_u32(smem);
  auto bar = [&](int i) -> uint32_t { return sb + OFF_BAR + 8u * (uint32_t)i; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_BAR + 96);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + OFF_BAR + 104);
  int* clamped = reinterpret_cast<int*>(smem + OFF_BAR + 108);
  volatile int* fix_any = reinterpret_cast<volatile int*>(smem + OFF_BAR + 112);
  float* sc = reinterpret_cast<float*>(smem + OFF_SC);
  float* sq = sc;                 // S_t / |p1_t|
  float* sk = sc + LT;            // S_t / |p2_t|
  float* s_self = sc + 2 * LT;    // S_t
  float* r1 = sc + 3 * LT;        // 1 / |p1_t|
  float* r2 = sc + 4 * LT;        // 1 / |p2_t|
  float* half_sum = sc + 5 * LT;  // [2][128]: per-channel sums of the two halves (log2 alpha,
                                  // then dL and Km Ys)
  float* lmid_s = sc + 7 * LT;    // [128] L_m per channel
  float* lend_s = sc + 8 * LT;    // [128] L_end per channel

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int blk = (int)(blockIdx.x % nb);
  const int bh = (int)(blockIdx.x / nb);  // one 64-column split per head at d_h = 64
  const int b = bh / p.H, h = bh % p.H;
  const int t0 = blk * LT;

  if (threadIdx.x == 0) {
    for (int i = 0; i < NBAR; ++i)
      mbar_init(bar(i), (i == B_OPS || i == B_A || i == B_DAS) ? 128 : 1);
    *abort_flag = 0;
    *clamped = 0;
    *fix_any = 0;
    fence_mbar_init();
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
      const uint32_t lb = bar(B_LOAD);
      mbar_arrive_expect_tx(lb, LOAD_BYTES);
      tma_load_4d(sb + OFF_P1, &tmP1, lb, 0, t0, h, b);
      tma_load_4d(sb + OFF_P2, &tmP2, lb, 0, t0, h, b);
      tma_load_4d(sb + OFF_V, &tmV, lb, 0, t0, h, b);
      tma_load_4d(sb + OFF_G, &tmG, lb, 0, t0, h, b);
      for (int k = 0; k < 2; ++k)
        tma_load_4d(sb + OFF_AL + k * LT * 128, &tmA, lb, k * 32, t0, h, b);
      tma_load_2d(sb + OFF_C0, &tmC0, lb, 0, (bh * (nb + 1) + blk) * D);
      tma_load_2d(sb + OFF_DC, &tmDC, lb, 0, (bh * nb + blk) * D);
      // p1 and p2 again (Qm and Km overwrote them) once the MMAs reading those are done
      bool ok = mbar_wait(bar(B_MM), 0, ab);
      if (ok) {
        mbar_arrive_expect_tx(bar(B_RELOAD), 2 * T16);
        tma_load_4d(sb + OFF_P1, &tmP1, bar(B_RELOAD), 0, t0, h, b);
        tma_load_4d(sb + OFF_P2, &tmP2, bar(B_RELOAD), 0, t0, h, b);
      }
      drain_wait(lb, 0);
      if (ok && ab.raised()) drain_wait(bar(B_RELOAD), 0);
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------------ MMA issuer
    constexpr uint32_t id_s = idesc_bf16_f32(128, 128, false, false);  // S, dA
    constexpr uint32_t id_kk = idesc_bf16_f32(128, 64, false, false);  // A, B K-major
    constexpr uint32_t id_km = idesc_bf16_f32(128, 64, false, true);   // B MN-major
    constexpr uint32_t id_mm = idesc_bf16_f32(128, 64, true, true);    // A, B MN-major
    bool ok = mbar_wait_warp(bar(B_OPS), 0, ab);
    if (ok) {
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)  // S = Qm Km^T  (K = 64 channels)
        mma_ss_w(tmem + COL_SC, smem_desc_sw128(sb + OFF_P1 + kk * 32, 16, 1024),
                 smem_desc_sw128(sb + OFF_P2 + kk * 32, 16, 1024), id_s, kk > 0 ? 1u : 0u);
      mma_commit_w(bar(B_S));
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)  // X = G (2^{L_m} C_0)^T   (K = 64 columns n)
        mma_ss_w(tmem + COL_X, smem_desc_sw128(sb + OFF_G + kk * 32, 16, 1024),
                 smem_desc_sw128(sb + OFF_C0 + kk * 32, 16, 1024), id_kk, kk > 0 ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)  // Ys = I~ (2^{L_end - L_m} dC)^T
        mma_ss_w(tmem + COL_YS, smem_desc_sw128(sb + OFF_V + kk * 32, 16, 1024),
                 smem_desc_sw128(sb + OFF_DCP + kk * 32, 16, 1024), id_kk, kk > 0 ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)  // dI~ = KL dC   (A = KL [j][c], B = dC [c][n] MN-major)
        mma_ss_w(tmem + COL_DI, smem_desc_sw128(sb + OFF_KL + kk * 32, 16, 1024),
                 smem_desc_sw128(sb + OFF_DC + kk * 16 * 128, 64 * 128, 1024), id_km,
                 kk > 0 ? 1u : 0u);
      ok = mbar_wait_warp(bar(B_A), 0, ab);  // A in shared memory, S read out
    }
    if (ok) {
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)  // dA = G I~^T   (N = 128 tokens j, K = 64 columns)
        mma_ss_w(tmem + COL_SC, smem_desc_sw128(sb + OFF_G + kk * 32, 16, 1024),
                 smem_desc_sw128(sb + OFF_V + kk * 32, 16, 1024), id_s, kk > 0 ? 1u : 0u);
      mma_commit_w(bar(B_DA));
#pragma unroll
      for (int kk = 0; kk < LT / 16; ++kk)  // dI~ += A^T G   (A^T: MN-major view of [t][j])
        mma_ss_w(tmem + COL_DI, smem_desc_sw128(sb + OFF_AS + kk * 16 * 128, LT * 128, 1024),
                 smem_desc_sw128(sb + OFF_G + kk * 16 * 128, LT * 128, 1024), id_mm, 1u);
      ok = mbar_wait_warp(bar(B_DAS), 0, ab);  // dA in shared memory
    }
    if (ok) {
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < LT / 16; ++kk) {  // X += dA Km   (K = 128 tokens j)
        const uint32_t koff = (kk >> 2) * (LT * 128) + (kk & 3) * 32;
        mma_ss_w(tmem + COL_X, smem_desc_sw128(sb + OFF_DAS + koff, 16, 1024),
                 smem_desc_sw128(sb + OFF_P2 + kk * 16 * 128, LT * 128, 1024), id_km, 1u);
      }
#pragma unroll
      for (int kk = 0; kk < LT / 16; ++kk)  // Y = dA^T Qm  (K = 128 tokens t)
        mma_ss_w(tmem + COL_Y, smem_desc_sw128(sb + OFF_DAS + kk * 16 * 128, LT * 128, 1024),
                 smem_desc_sw128(sb + OFF_P1 + kk * 16 * 128, LT * 128, 1024), id_mm,
                 kk > 0 ? 1u : 0u);
    }
    mma_commit_w(bar(B_MM));  // every product (or whatever completed before an abort)
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ elementwise
    const int t = threadIdx.x;  // token of the block / TMEM lane; channel c = t & 63, half
    const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
    const float inv_tau_sqrt_d = 1.0f / (p.tau_s * sqrtf((float)D));
    const int c = t & 63, half = t >> 6;
    uint8_t* const p1s = smem + OFF_P1;
    uint8_t* const p2s = smem + OFF_P2;
    float* const al = reinterpret_cast<float*>(smem + OFF_AL);
    auto al_at = [&](int tok, int ch) -> float& {  // [2][128][32] fp32, 128-byte swizzle
      return al[al_swz(tok, ch)];
    };
    float* const gl = reinterpret_cast<float*>(smem + OFF_GL);  // dL [t][GS]
    float* const ts = reinterpret_cast<float*>(smem + OFF_TS);  // Km Ys [t][GS]
    bool ok = true, my_clamp = false;
    do {
      ok = __all_sync(0xffffffffu, mbar_wait(bar(B_LOAD), 0, ab));
      if (!ok) break;
      // ---- phase A (thread = token): S_t, 1 / |p1_t|, 1 / |p2_t| (zero past T)
      {
        float dot = 0.f, n1 = 0.f, n2 = 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint32_t off = t * 128 + ((k ^ (t & 7)) << 4);
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
        float S = 0.f, i1 = 0.f, i2 = 0.f;
        if (t0 + t < p.T) {
          S = 1.0f / (1.0f + __expf(-dot * inv_tau_sqrt_d));
          i1 = rsqrtf(n1);
          i2 = rsqrtf(n2);
        }
        sq[t] = S * i1;
        sk[t] = S * i2;
        s_self[t] = S;
        r1[t] = i1;
        r2[t] = i2;
      }
      // ---- phase B, pass 1 (thread = channel and half block): running sums of log2 alpha
      // in place of alpha (the second half's relative to its start), 16 tokens ahead
      float lsum = 0.f;
      for (int i0 = 0; i0 < 64; i0 += 16) {
        float la[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          const int tok = half * 64 + i0 + u;
          la[u] = (t0 + tok < p.T) ? __log2f(al_at(tok, c)) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          lsum += la[u];
          al_at(half * 64 + i0 + u, c) = lsum;
        }
      }
      half_sum[half * 128 + c] = lsum;
      ew_sync();
      const float l_mid = half_sum[c], l_end = half_sum[c] + half_sum[128 + c];
      if (half == 0) {
        lmid_s[c] = l_mid;
        lend_s[c] = l_end;
        // C_0 scaled by 2^{L_m} in place, dC scaled by 2^{L_end - L_m} into its own tile
        // (row c; both factors <= 1)
        const float f0 = ex2_approx(l_mid), f1 = ex2_approx(l_end - l_mid);
        uint8_t* r0 = smem + OFF_C0 + c * 128;
        const uint8_t* rd = smem + OFF_DC + c * 128;
        uint8_t* rp = smem + OFF_DCP + c * 128;
#pragma unroll
        for (int k0 = 0; k0 < 8; ++k0) {
          const int k = (k0 + c) & 7;  // rows 128 bytes apart: rotate the 16-byte groups
          const uint4 a4 = *reinterpret_cast<const uint4*>(r0 + 16 * k);
          const uint4 d4 = *reinterpret_cast<const uint4*>(rd + 16 * k);
          const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w}, dw[4] = {d4.x, d4.y, d4.z, d4.w};
          uint32_t oa[4], od[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&aw[e]));
            const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&dw[e]));
            oa[e] = pack_bf16x2(x.x * f0, x.y * f0);
            od[e] = pack_bf16x2(y.x * f1, y.y * f1);
          }
          *reinterpret_cast<uint4*>(r0 + 16 * k) = make_uint4(oa[0], oa[1], oa[2], oa[3]);
          *reinterpret_cast<uint4*>(rp + 16 * k) = make_uint4(od[0], od[1], od[2], od[3]);
        }
      }
      ew_sync();
      // ---- phase B, pass 2 (thread = token): Qm, Km in place of p1, p2, and KL
      {
        const float s1 = sq[t], s2 = sk[t];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint32_t off = t * 128 + ((k ^ (t & 7)) << 4);
          const uint4 a4 = *reinterpret_cast<const uint4*>(p1s + off);
          const uint4 b4 = *reinterpret_cast<const uint4*>(p2s + off);
          const float4 L0 = *reinterpret_cast<const float4*>(&al_at(t, 8 * k));
          const float4 L1 = *reinterpret_cast<const float4*>(&al_at(t, 8 * k + 4));
          const float Lv[8] = {L0.x, L0.y, L0.z, L0.w, L1.x, L1.y, L1.z, L1.w};
          const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w}, bw[4] = {b4.x, b4.y, b4.z, b4.w};
          uint32_t qm[4], km[4], kl[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&aw[e]));
            const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bw[e]));
            float r[2][3];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
              const int ch = 8 * k + 2 * e + u;
              const float Lm = lmid_s[ch];
              const float L = Lv[2 * e + u] + (t >= 64 ? Lm : 0.f);
              const float dm = dm_of(Lv[2 * e + u], Lm, t >= 64, my_clamp);
              const float xv = u ? x.y : x.x, yv = u ? y.y : y.x;
              qm_km(xv, yv, s1, s2, dm, r[u][0], r[u][1]);
              r[u][2] = yv * s2 * ex2_approx(lend_s[ch] - L);       // KL (factor <= 1)
            }
            qm[e] = pack_bf16x2(r[0][0], r[1][0]);
            km[e] = pack_bf16x2(r[0][1], r[1][1]);
            kl[e] = pack_bf16x2(r[0][2], r[1][2]);
          }
          *reinterpret_cast<uint4*>(p1s + off) = make_uint4(qm[0], qm[1], qm[2], qm[3]);
          *reinterpret_cast<uint4*>(p2s + off) = make_uint4(km[0], km[1], km[2], km[3]);
          *reinterpret_cast<uint4*>(smem + OFF_KL + off) = make_uint4(kl[0], kl[1], kl[2], kl[3]);
        }
      }
      fence_async_smem();
      ew_sync();
      mbar_arrive(bar(B_OPS));
      // ---- phase D: A = tril(S, -1), then dA = tril(G I~^T, -1), as bf16 rows [t][j] in
      // shared memory (the products read them K-major and, transposed, MN-major)
      for (int pass = 0; pass < 2; ++pass) {
        ok = __all_sync(0xffffffffu, mbar_wait(bar(pass == 0 ? B_S : B_DA), 0, ab));
        if (!ok) break;
        tc_fence_after();
        uint8_t* dst = smem + (pass == 0 ? OFF_AS : OFF_DAS);
#pragma unroll
        for (int c0 = 0; c0 < LT; c0 += 32) {
          uint32_t s[32], pk[16];
          tmem_ld32(trow + COL_SC + c0, s);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            const float lo = (c0 + j < t) ? __uint_as_float(s[j]) : 0.f;
            const float hi = (c0 + j + 1 < t) ? __uint_as_float(s[j + 1]) : 0.f;
            pk[j >> 1] = pack_bf16x2(lo, hi);
          }
#pragma unroll
          for (int q = 0; q < 4; ++q)
            *reinterpret_cast<uint4*>(dst + swz(t, c0 + 8 * q, LT)) =
                make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
        }
        fence_async_smem();
        tc_fence_before();
        mbar_arrive(bar(pass == 0 ? B_A : B_DAS));
      }
      if (!ok) break;
      // ---- phase E (thread = token): every product done, p1 and p2 back in shared memory
      ok = __all_sync(0xffffffffu, mbar_wait(bar(B_MM), 0, ab) && mbar_wait(bar(B_RELOAD), 0, ab));
      if (!ok) break;
      tc_fence_after();
      {
        const float s1 = sq[t], s2 = sk[t], i1 = r1[t], i2 = r2[t], S = s_self[t];
        uint8_t* const gs = smem + OFF_G;
        bool unused_clamp = false;
        // channels [c0, c0 + 32): X, Y = dA^T Qm + Ys, Ys (and dI~) from TMEM
        auto load_xy = [&](int c0, uint32_t (&x)[32], uint32_t (&y)[32], uint32_t (&ys)[32],
                           uint32_t* di) {
          tmem_ld32(trow + COL_X + c0, x);
          tmem_ld32(trow + COL_Y + c0, y);
          tmem_ld32(trow + COL_YS + c0, ys);
          if (di) tmem_ld32(trow + COL_DI + c0, di);
          tmem_ld_wait();
        };
        // pass 1 (8 channels at a time): dq' = 2^{L_t - L_m} X, dk' = 2^{L_m - L_t} Y, the
        // dots p1 . dq' and p2 . dk', dL = Qm X - Km Y and Km Ys (Qm, Km as the products
        // read them), dv = dI~ + dY (in dY's place)
        float A1 = 0.f, A2 = 0.f;
#pragma unroll 1
        for (int c0 = 0; c0 < 64; c0 += 32) {
          uint32_t x[32], y[32], ys[32], di[32];
          load_xy(c0, x, y, ys, di);
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int kc = (c0 >> 3) + k;
            const uint32_t off = t * 128 + ((kc ^ (t & 7)) << 4);
            const uint4 a4 = *reinterpret_cast<const uint4*>(p1s + off);
            const uint4 b4 = *reinterpret_cast<const uint4*>(p2s + off);
            const uint4 g4 = *reinterpret_cast<const uint4*>(gs + off);
            const float4 L0 = *reinterpret_cast<const float4*>(&al_at(t, 8 * kc));
            const float4 L1 = *reinterpret_cast<const float4*>(&al_at(t, 8 * kc + 4));
            const float Lv[8] = {L0.x, L0.y, L0.z, L0.w, L1.x, L1.y, L1.z, L1.w};
            const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w}, bw[4] = {b4.x, b4.y, b4.z, b4.w},
                           gw[4] = {g4.x, g4.y, g4.z, g4.w};
            float dl[8], tv[8];
            uint32_t dvw[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 xa = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&aw[e]));
              const float2 yb = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bw[e]));
              const float2 g = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&gw[e]));
              float dvv[2];
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int j = 8 * k + 2 * e + u;  // index within the 32 loaded columns
                const int ch = 8 * kc + 2 * e + u;
                const float pv = u ? xa.y : xa.x, kv = u ? yb.y : yb.x;
                const float dm = dm_of(Lv[2 * e + u], lmid_s[ch], t >= 64, unused_clamp);
                float qm, km;
                qm_km(pv, kv, s1, s2, dm, qm, km);
                const float X = __uint_as_float(x[j]), Ysv = __uint_as_float(ys[j]);
                const float Y = __uint_as_float(y[j]) + Ysv;
                A1 = fmaf(pv, ex2_approx(dm) * X, A1);
                A2 = fmaf(kv, ex2_approx(-dm) * Y, A2);
                dl[2 * e + u] = qm * X - km * Y;
                tv[2 * e + u] = km * Ysv;
                dvv[u] = __uint_as_float(di[j]) + (u ? g.y : g.x);
              }
              dvw[e] = pack_bf16x2(dvv[0], dvv[1]);
            }
            *reinterpret_cast<uint4*>(gs + off) = make_uint4(dvw[0], dvw[1], dvw[2], dvw[3]);
            float* gr = gl + t * GS + 8 * kc;
            *reinterpret_cast<float4*>(gr) = make_float4(dl[0], dl[1], dl[2], dl[3]);
            *reinterpret_cast<float4*>(gr + 4) = make_float4(dl[4], dl[5], dl[6], dl[7]);
            float* tr = ts + t * GS + 8 * kc;
            *reinterpret_cast<float4*>(tr) = make_float4(tv[0], tv[1], tv[2], tv[3]);
            *reinterpret_cast<float4*>(tr + 4) = make_float4(tv[4], tv[5], tv[6], tv[7]);
          }
        }
        // pass 2: through S_t and the normalisation of p1, p2 (written in their place)
        //   dp1 = S/|p1| dq' - S/|p1|^3 (p1 . dq') p1 + du p2, and symmetrically dp2,
        //   du = (p1 . dq' / |p1| + p2 . dk' / |p2|) S (1 - S) / (tau_S sqrt(d_h))
        const float du = (i1 * A1 + i2 * A2) * S * (1.0f - S) * inv_tau_sqrt_d;
        const float c1 = s1 * i1 * i1 * A1, c2 = s2 * i2 * i2 * A2;
#pragma unroll 1
        for (int c0 = 0; c0 < 64; c0 += 32) {
          uint32_t x[32], y[32], ys[32];
          load_xy(c0, x, y, ys, nullptr);
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int kc = (c0 >> 3) + k;
            const uint32_t off = t * 128 + ((kc ^ (t & 7)) << 4);
            const uint4 a4 = *reinterpret_cast<const uint4*>(p1s + off);
            const uint4 b4 = *reinterpret_cast<const uint4*>(p2s + off);
            const float4 L0 = *reinterpret_cast<const float4*>(&al_at(t, 8 * kc));
            const float4 L1 = *reinterpret_cast<const float4*>(&al_at(t, 8 * kc + 4));
            const float Lv[8] = {L0.x, L0.y, L0.z, L0.w, L1.x, L1.y, L1.z, L1.w};
            const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w}, bw[4] = {b4.x, b4.y, b4.z, b4.w};
            uint32_t o1[4], o2[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 xa = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&aw[e]));
              const float2 yb = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bw[e]));
              float r1v[2], r2v[2];
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int j = 8 * k + 2 * e + u;
                const int ch = 8 * kc + 2 * e + u;
                const float pv = u ? xa.y : xa.x, kv = u ? yb.y : yb.x;
                const float dm = dm_of(Lv[2 * e + u], lmid_s[ch], t >= 64, unused_clamp);
                const float dq = ex2_approx(dm) * __uint_as_float(x[j]);
                const float dk = ex2_approx(-dm) * (__uint_as_float(y[j]) + __uint_as_float(ys[j]));
                r1v[u] = fmaf(s1, dq, fmaf(-c1, pv, du * kv));
                r2v[u] = fmaf(s2, dk, fmaf(-c2, kv, du * pv));
              }
              o1[e] = pack_bf16x2(r1v[0], r1v[1]);
              o2[e] = pack_bf16x2(r2v[0], r2v[1]);
            }
            *reinterpret_cast<uint4*>(p1s + off) = make_uint4(o1[0], o1[1], o1[2], o1[3]);
            *reinterpret_cast<uint4*>(p2s + off) = make_uint4(o2[0], o2[1], o2[2], o2[3]);
          }
        }
        fence_async_smem();
        __syncwarp();
        if (lane == 0 && t0 + warp * 32 < p.T) {  // this warp's 32 rows of dp1, dp2, dv
          const uint32_t so = (uint32_t)warp * (32 * 128);
          tma_store_4d(&tmDP1, sb + OFF_P1 + so, 0, t0 + warp * 32, h, b);
          tma_store_4d(&tmDP2, sb + OFF_P2 + so, 0, t0 + warp * 32, h, b);
          tma_store_4d(&tmDV, sb + OFF_G + so, 0, t0 + warp * 32, h, b);
          tma_store_commit();
        }
      }
      // ---- phase F (thread = channel and half block): dalpha_u = (end + sum_{t >= u} dL_t)
      // / alpha_u, end = sum_n (2^{L_m} C_0)[c][n] (2^{L_end - L_m} dC)[c][n] + sum_j Km_j Ys_j
      ew_sync();
      {
        float e0 = 0.f;
        const uint8_t* rc0 = smem + OFF_C0 + c * 128;
        const uint8_t* rdp = smem + OFF_DCP + c * 128;
#pragma unroll
        for (int k0 = 0; k0 < 8; ++k0) {  // same swizzle in both tiles: a plain row dot
          const int k = (k0 + c) & 7;     // rows 128 bytes apart: rotate the 16-byte groups
          const uint4 a4 = *reinterpret_cast<const uint4*>(rc0 + 16 * k);
          const uint4 d4 = *reinterpret_cast<const uint4*>(rdp + 16 * k);
          const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w}, dw[4] = {d4.x, d4.y, d4.z, d4.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&aw[e]));
            const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&dw[e]));
            e0 = fmaf(x.x, y.x, fmaf(x.y, y.y, e0));
          }
        }
        float glh = 0.f, tsh = 0.f;
#pragma unroll
        for (int i0 = 0; i0 < 64; i0 += 16) {  // 16 independent loads in flight
          float g16[16], t16[16];
#pragma unroll
          for (int u = 0; u < 16; ++u) {
            g16[u] = gl[(half * 64 + i0 + u) * GS + c];
            t16[u] = ts[(half * 64 + i0 + u) * GS + c];
          }
#pragma unroll
          for (int u = 0; u < 16; ++u) {
            glh += g16[u];
            tsh += t16[u];
          }
        }
        half_sum[half * 128 + c] = glh;
        half_sum[half * 128 + 64 + c] = tsh;
        ew_sync();
        // what the block's end and (for the first half) the later half carry
        float run = e0 + half_sum[64 + c] + half_sum[128 + 64 + c] +
                    (half == 0 ? half_sum[128 + c] : 0.f);
        const float* arow = p.alpha + (long long)b * p.sB + (long long)h * p.sH + c;
        float* drow = p.dalpha + (long long)b * p.sB + (long long)h * p.sH + c;
        unsigned long long small = 0ull;  // tokens of the half with alpha < kSmallAlpha
        for (int i0 = 48; i0 >= 0; i0 -= 16) {  // 16 tokens: loads first, then the suffix
          float a16[16], g16[16];
#pragma unroll
          for (int u = 0; u < 16; ++u) {
            const int tok = half * 64 + i0 + u;
            a16[u] = t0 + tok < p.T ? __ldg(arow + (long long)(t0 + tok) * p.sT) : 1.f;
            g16[u] = gl[tok * GS + c];
          }
#pragma unroll
          for (int u = 15; u >= 0; --u) {
            const int tok = half * 64 + i0 + u;
            run += g16[u];
            if (t0 + tok < p.T) drow[(long long)(t0 + tok) * p.sT] = run / a16[u];
            if (a16[u] < kSmallAlpha) small |= 1ull << (i0 + u);
          }
        }
        // A small alpha_u (below 2^-10) leaves the suffix sum above a small remainder of
        // terms that cancel, whose fp32 rounding the division magnifies.  There dalpha comes
        // from the state entering u and the adjoint of Diag(alpha_u) C_{u-1}, channel c (row
        // c), at the midpoint scale:
        //   P_u = 2^{L_m} C_0 + sum_{j < u} Km_j I~_j,   Q_u = 2^{L_end - L_m} dC + sum_{t >= u} Qm_t dY_t,
        //   dalpha_u = <P_u, Q_u> / alpha_u,
        // where every term of P_u (u in the first half) or of Q_u (the second) carries the
        // factor alpha_u, so nothing large cancels.  A block with such tokens loads dY, p1
        // and p2 again (their tiles now hold the outputs) over the dL arrays, which every
        // elementwise warp has read by then; one warp per (u, c), Km and Qm in fp32.
        const bool warp_small = small_any_warp(small);  // every lane takes part in the vote
        if (lane == 0 && warp_small) *fix_any = 1;
        ew_sync();
        if (*fix_any) {
          if (threadIdx.x == 0) {
            fence_async_smem();  // the dL arrays' generic accesses precede the copies
            mbar_arrive_expect_tx(bar(B_FIX), 3 * T16);
            tma_load_4d(sb + OFF_FIX_G, &tmG, bar(B_FIX), 0, t0, h, b);
            tma_load_4d(sb + OFF_FIX_P1, &tmP1, bar(B_FIX), 0, t0, h, b);
            tma_load_4d(sb + OFF_FIX_P2, &tmP2, bar(B_FIX), 0, t0, h, b);
          }
          if (!(ok = __all_sync(0xffffffffu, mbar_wait(bar(B_FIX), 0, ab)))) break;
          const uint8_t* vt = smem + OFF_V;
          const uint8_t* gt = smem + OFF_FIX_G;
          const uint8_t* p1t = smem + OFF_FIX_P1;
          const uint8_t* p2t = smem + OFF_FIX_P2;
          const uint8_t* c0t = smem + OFF_C0;
          const uint8_t* dct = smem + OFF_DCP;
          const int t_live = min(LT, p.T - t0);
          bool unused_clamp = false;
          // lanes: token group g4 (tokens = g4 mod 4) and the 8 columns from nc (16-byte
          // group lane & 7 of a 128-byte swizzled row)
          const int g4 = lane >> 3;
          auto row16 = [&](const uint8_t* tile, int r) {
            return *reinterpret_cast<const uint4*>(
                tile + r * 128 + ((((uint32_t)lane & 7) ^ ((uint32_t)r & 7)) << 4));
          };
          auto elem = [&](const uint8_t* tile, int r, int col) {
            return __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(
                tile + r * 128 + ((((uint32_t)col >> 3) ^ ((uint32_t)r & 7)) << 4) + (col & 7) * 2));
          };
          for (int i = 0; i < 64 && warp_small; ++i) {
            unsigned fl = __ballot_sync(0xffffffffu, ((small >> i) & 1ull) != 0ull);
            while (fl) {
              const int src = __ffs(fl) - 1;
              fl &= fl - 1;
              const int cc = (warp & 1) * 32 + src;  // that lane's channel
              const int u = half * 64 + i;
              const float lmc = lmid_s[cc];
              // Km of the tokens before u and Qm of those from u on, channel cc: lane l
              // holds tokens l + 32 k
              float kmr[4], qmr[4];
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const int tok = lane + 32 * k;
                const float dm = dm_of(al_at(tok, cc), lmc, tok >= 64, unused_clamp);
                const float x2 = tok < u ? elem(p2t, tok, cc) : 0.f;
                const float x1 = (tok >= u && tok < t_live) ? elem(p1t, tok, cc) : 0.f;
                kmr[k] = x2 * sk[tok] * ex2_approx(-dm);
                qmr[k] = x1 * sq[tok] * ex2_approx(dm);
              }
              float P[8], Q[8];
#pragma unroll
              for (int e = 0; e < 8; ++e) P[e] = Q[e] = 0.f;
#pragma unroll 4
              for (int j0 = 0; j0 < LT; j0 += 4) {  // tokens j0 + g4
                const int j = j0 + g4, kq = j0 >> 5;
                const float ksel = kq == 0 ? kmr[0] : kq == 1 ? kmr[1] : kq == 2 ? kmr[2] : kmr[3];
                const float qsel = kq == 0 ? qmr[0] : kq == 1 ? qmr[1] : kq == 2 ? qmr[2] : qmr[3];
                const float km = __shfl_sync(0xffffffffu, ksel, (j0 & 31) + g4);
                const float qm = __shfl_sync(0xffffffffu, qsel, (j0 & 31) + g4);
                const uint4 v4 = row16(vt, j), d4 = row16(gt, j);
                const uint32_t vw[4] = {v4.x, v4.y, v4.z, v4.w}, dw[4] = {d4.x, d4.y, d4.z, d4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const float2 fv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&vw[e]));
                  const float2 fd = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&dw[e]));
                  P[2 * e] = fmaf(km, fv.x, P[2 * e]);
                  P[2 * e + 1] = fmaf(km, fv.y, P[2 * e + 1]);
                  Q[2 * e] = fmaf(qm, fd.x, Q[2 * e]);
                  Q[2 * e + 1] = fmaf(qm, fd.y, Q[2 * e + 1]);
                }
              }
              // the four token groups' sums, the block-boundary rows, and <P_u, Q_u>
              const uint4 c4 = row16(c0t, cc), e4 = row16(dct, cc);
              const uint32_t cw[4] = {c4.x, c4.y, c4.z, c4.w}, ew[4] = {e4.x, e4.y, e4.z, e4.w};
              float pq = 0.f;
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float2 cf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&cw[e]));
                const float2 ef = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ew[e]));
#pragma unroll
                for (int h2 = 0; h2 < 2; ++h2) {
                  float pe = P[2 * e + h2], qe = Q[2 * e + h2];
                  pe += __shfl_xor_sync(0xffffffffu, pe, 8);
                  pe += __shfl_xor_sync(0xffffffffu, pe, 16);
                  qe += __shfl_xor_sync(0xffffffffu, qe, 8);
                  qe += __shfl_xor_sync(0xffffffffu, qe, 16);
                  pq = fmaf(pe + (h2 ? cf.y : cf.x), qe + (h2 ? ef.y : ef.x), pq);
                }
              }
              pq += __shfl_xor_sync(0xffffffffu, pq, 1);
              pq += __shfl_xor_sync(0xffffffffu, pq, 2);
              pq += __shfl_xor_sync(0xffffffffu, pq, 4);
              if (lane == src)
                drow[(long long)(t0 + u) * p.sT] = pq / __ldg(arow + (long long)(t0 + u) * p.sT);
            }
          }
        }
      }
    } while (false);
    if (lane == 0) tma_store_wait_read_all();
    if (my_clamp) atomicExch(clamped, 1);
  }

  if (warp == 5) drain_wait(bar(B_MM), 0);  // no product in flight past the teardown
  if (threadIdx.x == 0 && *fix_any) drain_wait(bar(B_FIX), 0);  // nor the fix-up's copies
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *clamped && p.dev_status && !*abort_flag)
    atomicExch(p.dev_status, (int)RELATION_ERR_UNSUPPORTED);
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace bwd
}  // namespace lintc

bool linear_tc_bwd_supports(const LinearProblem& p) {
  return p.dtype == RELATION_BF16 && p.d == 64 && p.sB % 8 == 0 && p.sT % 8 == 0 &&
         p.sH % 8 == 0;
}

size_t linear_tc_bwd_workspace_bytes(const LinearProblem& p) {
  if (!linear_tc_bwd_supports(p)) return 0;
  const long long heads = (long long)p.B * p.H, nb = (p.T + lintc::LT - 1) / lintc::LT;
  return lintc::bwd_bytes(heads, nb, 64, nullptr, nullptr, nullptr);
}

// Five launches: the four state passes (states_t), then one CTA per (head, block).
cudaError_t launch_linear_tc_bwd(const LinearProblem& p, cudaStream_t s) {
  using namespace lintc;
  if (!linear_tc_bwd_supports(p) || !p.workspace) return cudaErrorInvalidValue;
  const int nb = (p.T + LT - 1) / LT;
  const long long heads = (long long)p.B * p.H;
  const long long grid = heads * nb;
  if (grid > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(bwd::lin_tc_bwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                bwd::SMEM)) != cudaSuccess) {
    note_failure("linear chunked backward: shared memory attribute");
    return e;
  }
  if ((e = states_t<64>(p, p.dy, p.workspace, s)) != cudaSuccess) return e;
  LinCp cp{};
  __nv_bfloat16* dcb = nullptr;
  bwd_bytes(heads, nb, 64, &cp, &dcb, p.workspace);
  Problem q{};  // the bf16 tensor-map helper's view of the shapes
  q.B = p.B; q.T = p.T; q.H = p.H; q.d = p.d;
  q.sB = p.sB; q.sT = p.sT; q.sH = p.sH;
  CUtensorMap m1, m2, mv, mg, ma, mc0, mdc, o1, o2, ov;
  if (!tc::make_tmap_bf16(&m1, p.p1, q, LT) || !tc::make_tmap_bf16(&m2, p.p2, q, LT) ||
      !tc::make_tmap_bf16(&mv, p.v, q, LT) || !tc::make_tmap_bf16(&mg, p.dy, q, LT) ||
      !make_tmap_alpha(&ma, p, true) || !make_tmap_c0(&mc0, cp.c0, heads * (nb + 1) * 64, 64) ||
      !make_tmap_c0(&mdc, dcb, heads * nb * 64, 64) || !tc::make_tmap_bf16(&o1, p.dp1, q, 32) ||
      !tc::make_tmap_bf16(&o2, p.dp2, q, 32) || !tc::make_tmap_bf16(&ov, p.dv, q, 32)) {
    note_failure("linear chunked backward: TMA descriptors");
    return cudaErrorInvalidValue;
  }
  bwd::lin_tc_bwd_kernel<<<(unsigned)grid, kThreads, bwd::SMEM, s>>>(m1, m2, mv, mg, ma, mc0, mdc,
                                                                    o1, o2, ov, p, nb);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("linear chunked backward: launch");
  return e;
}

}  // namespace rel
