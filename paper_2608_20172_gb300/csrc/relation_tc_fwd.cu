// relation_tc_fwd.cu -- tcgen05 / TMA / TMEM forward of FlashRelation (bf16, d_h 64 or 128).
//
// One CTA owns a tile of BM = 128 query rows of one head and scans the key/value tiles
// j0 = 0, 128, ... up to and including its diagonal tile (Sec. 5.1, App. A.3).  Several
// CTAs share an SM (d_h = 128: two of 256 TMEM columns; d_h = 64: four of 128), so the
// tensor core of one CTA overlaps the elementwise work of the others.  CTAs take the
// heaviest query tiles first, heads in groups (grouped_unit), so that the K/V rows in use
// stay in L2.
//
// Warp roles (192 threads):
//   warps 0-3  Exchange scan + epilogue: thread t owns query row q0 + t (TMEM lane t).
//   warp  4    TMA producer: Q tile once, then K and V through a ring of stages.
//   warp  5    TMEM allocator and MMA issuer (one elected thread).
// The scan advances SK keys per step (64 at d_h = 128, 32 at d_h = 64) through two TMEM
// buffers, so the MMAs of one step (U of step s + 2, z += P V of step s) overlap the
// elementwise work of the next.  Step s:
//   MMA   U = Q K^T over SK keys                -> TMEM columns [SK b, SK b + SK), b = s & 1
//   scan  E = SiLU(U / sqrt(d)) for keys < row (Self excluded); P = exp(E - m) at the row's
//         scale m (an upper bound of max E, max(U, 0) / sqrt(d), raised a step late when
//         it grew by > 2^8), row sum l += sum P; P as bf16 written back into the buffer's
//         first SK / 2 columns (two per 32-bit column); the diagonal tile also yields
//         S_i = sigmoid(U_ii / (sqrt(d) tau_S)).
//   MMA   z += P V  (A operand P read from TMEM)  -> TMEM columns [2 SK, 2 SK + d)
// Epilogue (App. A.3.3-A.3.5): L^E = m + log l, A = L^E - lambda log i,
//   g = sigmoid(A - S), Y = (1 - g) v_i + g z / l, logZ = logaddexp(S, A); row 1 has an
//   empty history: g = 0, Y = v_1, logZ = S_1 (App. A.1.8).
// R and F never leave the SM.  Every mbarrier wait is bounded (common.cuh).
#include <cudaTypedefs.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace rel {
namespace tc {

constexpr int BM = 128;        // query rows per CTA
constexpr int BN = 128;        // keys per K/V tile (TMA granularity)
constexpr int HN = 64;         // half a K/V tile: the register scan's step, the d_h = 64 load
constexpr int kSCol = 0;       // U/P buffer b at kSCol + SK b
constexpr float kRescaleLog2 = 8.0f;  // rescale z only when the max grows by > 2^8
constexpr float kStaleLog2 = 32.0f;   // a step's P may reach 2^32 at the previous scale

// d_h = 64 (QUAD): four CTAs per SM, so that each SM sub-partition runs four scan warps:
//   TMEM 128 columns (two U/P buffers of 32-key steps + z 64), K and V in 64-key halves
//   through two stages each (50 KB of shared memory).
// d_h = 128: two CTAs per SM, two U/P buffers of 64-key steps (so that the MMAs of one step
//   overlap the scan of the next) + z 128 = 256 TMEM columns, 128-key K/V tiles through one
//   stage.  (WIDE, steps of a whole 128-key tile in one buffer of 128 columns so that
//   U = Q K^T runs at N = 128, measured slower on the long workload, 2.40 against 1.98 ms:
//   each step then waits for its own 1024 cycles of MMAs, which two CTAs do not cover.)
// With one U/P buffer the scan takes a step in chunks of 32 keys (registers).
template <int D>
struct FwdCfg {
  static constexpr bool QUAD = D == 64;
  static constexpr bool WIDE = false;
  // DEEP: four buffers of 32-key steps (U three steps ahead) in the same 256 columns;
  // measured slower at d_h = 128 (long forward 1.97 -> 2.35 ms: U = Q K^T at N = 32 reads
  // the Q tile from shared memory twice as often per key)
  static constexpr bool DEEP = false;
  static constexpr int SK = WIDE ? 128 : ((QUAD || DEEP) ? 32 : HN);  // keys per scan step
  static constexpr int CTAS = QUAD ? 4 : 2;      // CTAs per SM
  static constexpr int TMEM_COLS = QUAD ? 128 : 256;
  static constexpr int NBUF = WIDE ? 1 : (DEEP ? 4 : 2);  // U/P buffers
  static constexpr int OCOL = NBUF * SK;         // z accumulator
  static constexpr int W_TMA = 4, W_MMA = 5;
  static constexpr int THREADS = 192;
  static constexpr int KB = D / 64;              // 64-column (128-byte) swizzle blocks along d
  static constexpr int TILE = BN * D * 2;        // bytes of the Q tile
  static constexpr int KVR = QUAD ? HN : BN;     // K / V rows per load (SK or 2 SK)
  static constexpr int KVT = KVR * D * 2;        // bytes of one K or V load
  static constexpr int STAGES = QUAD ? 2 : 1;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + TILE;
  static constexpr int OFF_V = OFF_K + STAGES * KVT;
  static constexpr int OFF_BAR = OFF_V + STAGES * KVT;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;  // barriers + 1024-byte alignment slack
  static_assert(CTAS * (SMEM + 1024) <= 233472, "CTAs per SM");
  static_assert(OCOL + D <= TMEM_COLS, "TMEM");
};

// mbarrier slots
enum : int {
  // per stage (2): B_KF .. B_VE; per U/P buffer (up to 4): B_S, B_P and B_OD (the z update
  // of a step of that buffer done, so that a wait for step s - 1's update is exact for any
  // number of buffers: U of step s implies the buffer's previous update)
  B_Q = 0, B_KF = 1, B_KE = 3, B_VF = 5, B_VE = 7, B_S = 9, B_P = 13, B_OD = 17, B_O = 21,
  NBAR_FWD = 22
};

// Bounded wait used while draining at teardown: never raises, just gives up.
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > 20ull * 1000ull * 1000ull) return;  // 20 ms
  }
}

__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Maximum of the raw evidence U over the row's history in one step; on the diagonal tile
// only the keys before the row's own (t, relative to the step's first key) count, and U at
// key t (the Self evidence U_ii) is returned in u_self.
template <bool DIAG>
__device__ __forceinline__ float row_max(const uint32_t (&U)[HN], int t, float& u_self) {
  if (!DIAG) {
    float m0 = __uint_as_float(U[0]), m1 = __uint_as_float(U[1]);
    float m2 = __uint_as_float(U[2]), m3 = __uint_as_float(U[3]);
#pragma unroll
    for (int c = 4; c + 8 <= HN; c += 8) {
      m0 = fmax3(m0, __uint_as_float(U[c]), __uint_as_float(U[c + 1]));
      m1 = fmax3(m1, __uint_as_float(U[c + 2]), __uint_as_float(U[c + 3]));
      m2 = fmax3(m2, __uint_as_float(U[c + 4]), __uint_as_float(U[c + 5]));
      m3 = fmax3(m3, __uint_as_float(U[c + 6]), __uint_as_float(U[c + 7]));
    }
    // the last four keys (the loop covers keys 4 .. HN - 5)
    m0 = fmax3(m0, __uint_as_float(U[HN - 4]), __uint_as_float(U[HN - 3]));
    m1 = fmax3(m1, __uint_as_float(U[HN - 2]), __uint_as_float(U[HN - 1]));
    return fmaxf(fmax3(m0, m1, m2), m3);
  }
  float m = -INFINITY;
#pragma unroll
  for (int c = 0; c < HN; ++c) {
    const float x = __uint_as_float(U[c]);
    m = c < t ? fmaxf(m, x) : m;
    u_self = c == t ? x : u_self;
  }
  return m;
}

// P = 2^(U c2k (1 + tanh(U ch)) - m) for the 64 keys of a step (0 off the history on the
// diagonal tile), written to TMEM columns pcol.. as bf16 pairs; returns the row sum as two
// halves, and on the way the maximum of the raw evidence over the row's history in the
// step (umax) and, on the diagonal tile, U_ii (u_self).
template <bool DIAG>
__device__ __forceinline__ float2 scan_p(const uint32_t (&U)[HN], int t, uint32_t pcol, float ch,
                                         float c2k, float negm, float& umax, float& u_self) {
  const float2 ch2 = make_float2(ch, ch), c2k2 = make_float2(c2k, c2k);
  const float2 nm2 = make_float2(negm, negm);
  float2 sum = make_float2(0.f, 0.f);
  float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
  for (int c0 = 0; c0 < HN; c0 += 32) {
    uint32_t pk[16];
#pragma unroll
    for (int c = 0; c < 32; c += 2) {
      const float2 x = make_float2(__uint_as_float(U[c0 + c]), __uint_as_float(U[c0 + c + 1]));
      const float2 h = __fmul2_rn(x, ch2);
      const float2 th = make_float2(tanh_approx(h.x), tanh_approx(h.y));
      const float2 w = __ffma2_rn(th, c2k2, c2k2);  // log2(e) sigma(u) / sqrt(d), times 2
      const float2 e = __ffma2_rn(x, w, nm2);
      float2 pv = make_float2(ex2_approx(e.x), ex2_approx(e.y));
      if (DIAG) {
        const bool in0 = c0 + c < t, in1 = c0 + c + 1 < t;
        pv.x = in0 ? pv.x : 0.f;
        pv.y = in1 ? pv.y : 0.f;
        mx0 = fmax3(mx0, in0 ? x.x : -INFINITY, in1 ? x.y : -INFINITY);
        u_self = c0 + c == t ? x.x : (c0 + c + 1 == t ? x.y : u_self);
      } else {
        (c & 2 ? mx1 : mx0) = fmax3(c & 2 ? mx1 : mx0, x.x, x.y);
      }
      sum = __fadd2_rn(sum, pv);
      pk[c >> 1] = pack_bf16x2(pv.x, pv.y);
    }
    tmem_st16(pcol + (c0 >> 1), pk);
  }
  umax = fmaxf(mx0, mx1);
  return sum;
}

// The four-CTA layout's scan works on 32 keys at a time (registers): the maximum of the
// raw evidence over the history among them (keys before t, relative to their first key,
// on a masked step), and U at key t in u_self.
template <bool DIAG>
__device__ __forceinline__ float row_max32(const uint32_t (&U)[32], int t, float& u_self) {
  if (!DIAG) {
    float m0 = __uint_as_float(U[0]), m1 = __uint_as_float(U[1]);
    float m2 = __uint_as_float(U[2]), m3 = __uint_as_float(U[3]);
#pragma unroll
    for (int c = 4; c + 8 <= 32; c += 8) {
      m0 = fmax3(m0, __uint_as_float(U[c]), __uint_as_float(U[c + 1]));
      m1 = fmax3(m1, __uint_as_float(U[c + 2]), __uint_as_float(U[c + 3]));
      m2 = fmax3(m2, __uint_as_float(U[c + 4]), __uint_as_float(U[c + 5]));
      m3 = fmax3(m3, __uint_as_float(U[c + 6]), __uint_as_float(U[c + 7]));
    }
    m0 = fmax3(m0, __uint_as_float(U[28]), __uint_as_float(U[29]));
    m1 = fmax3(m1, __uint_as_float(U[30]), __uint_as_float(U[31]));
    return fmaxf(fmax3(m0, m1, m2), m3);
  }
  float m = -INFINITY;
#pragma unroll
  for (int c = 0; c < 32; ++c) {
    const float x = __uint_as_float(U[c]);
    m = c < t ? fmaxf(m, x) : m;
    u_self = c == t ? x : u_self;
  }
  return m;
}

// P of 32 keys as 16 bf16 pairs (not stored), their row sum, and on the way the maximum
// of their raw evidence over the history and U_ii (as scan_p).
template <bool DIAG>
__device__ __forceinline__ float2 scan_p32(const uint32_t (&U)[32], int t, float ch, float c2k,
                                           float negm, float& umax, float& u_self,
                                           uint32_t (&pk)[16]) {
  const float2 ch2 = make_float2(ch, ch), c2k2 = make_float2(c2k, c2k);
  const float2 nm2 = make_float2(negm, negm);
  float2 sum = make_float2(0.f, 0.f);
  float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
  for (int c = 0; c < 32; c += 2) {
    const float2 x = make_float2(__uint_as_float(U[c]), __uint_as_float(U[c + 1]));
    const float2 h = __fmul2_rn(x, ch2);
    const float2 th = make_float2(tanh_approx(h.x), tanh_approx(h.y));
    const float2 w = __ffma2_rn(th, c2k2, c2k2);
    const float2 e = __ffma2_rn(x, w, nm2);
    float2 pv = make_float2(ex2_approx(e.x), ex2_approx(e.y));
    if (DIAG) {
      const bool in0 = c < t, in1 = c + 1 < t;
      pv.x = in0 ? pv.x : 0.f;
      pv.y = in1 ? pv.y : 0.f;
      mx0 = fmax3(mx0, in0 ? x.x : -INFINITY, in1 ? x.y : -INFINITY);
      u_self = c == t ? x.x : (c + 1 == t ? x.y : u_self);
    } else {
      (c & 2 ? mx1 : mx0) = fmax3(c & 2 ? mx1 : mx0, x.x, x.y);
    }
    sum = __fadd2_rn(sum, pv);
    pk[c >> 1] = pack_bf16x2(pv.x, pv.y);
  }
  umax = fmaxf(mx0, mx1);
  return sum;
}

// MODE 0: the forward (epilogue: Y, logZ, F_ii).  MODE 1: the Exchange summary only
// (st.m, st.l, st.z), over the queries' own earlier tokens (st.causal) or over every key
// of k, v (st.Tk of them, all preceding the queries; the ragged last tile masked).
template <int D, int MODE>
__global__ void __launch_bounds__(FwdCfg<D>::THREADS, FwdCfg<D>::CTAS)
    fwd_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO,
                  Problem p, int n_qt, int n_groups, StateArgs sa) {
  using C = FwdCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sb = smem_u32(smem);
  auto bar = [&](int i) -> uint32_t { return sb + C::OFF_BAR + 8u * (uint32_t)i; };
  static_assert(NBAR_FWD * 8 <= 192, "barrier slots");
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_BAR + 192);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_BAR + 200);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int BH = p.B * p.H;
  int tq, bh;  // heaviest query tiles first, heads in groups (common.cuh)
  grouped_unit((int)blockIdx.x, n_qt, BH, n_groups, tq, bh);
  const int qt = n_qt - 1 - tq;
  const int b = bh / p.H, h = bh % p.H;
  const int q0 = qt * BM;
  const bool causal = MODE == 0 || sa.causal;
  const int n_kv = causal ? qt + 1 : (sa.Tk + BN - 1) / BN;

  if (threadIdx.x == 0) {
    mbar_init(bar(B_Q), 1);
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(bar(B_KF + s), 1);
      mbar_init(bar(B_KE + s), 1);
      mbar_init(bar(B_VF + s), 1);
      mbar_init(bar(B_VE + s), 1);
    }
    for (int bb = 0; bb < C::NBUF; ++bb) {
      mbar_init(bar(B_S + bb), 1);
      mbar_init(bar(B_P + bb), 128);
      mbar_init(bar(B_OD + bb), 1);
    }
    mbar_init(bar(B_O), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == C::W_MMA) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const Abort ab{abort_flag, p.dev_status};

  if (warp == C::W_TMA) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      mbar_arrive_expect_tx(bar(B_Q), C::TILE);
      for (int kb = 0; kb < C::KB; ++kb)
        tma_load_4d(sb + C::OFF_Q + kb * BM * 128, &tmQ, bar(B_Q), kb * 64, q0, h, b);
      // K and V through the stage ring, one load unit (QUAD: a 64-key half, one scan step;
      // else a 128-key tile, two steps) at a time
      const int n_ld = n_kv * (BN / C::KVR);
      int issued = 0;
      for (int j = 0; j < n_ld; ++j) {
        const int s = j % C::STAGES, u = j / C::STAGES;
        if (u > 0 && !mbar_wait(bar(B_KE + s), (u - 1) & 1, ab)) break;
        mbar_arrive_expect_tx(bar(B_KF + s), C::KVT);
        for (int kb = 0; kb < C::KB; ++kb)
          tma_load_4d(sb + C::OFF_K + s * C::KVT + kb * C::KVR * 128, &tmK, bar(B_KF + s),
                      kb * 64, j * C::KVR, h, b);
        if (u > 0 && !mbar_wait(bar(B_VE + s), (u - 1) & 1, ab)) {
          issued = j + 1;  // K of unit j is in flight, V is not
          break;
        }
        mbar_arrive_expect_tx(bar(B_VF + s), C::KVT);
        for (int kb = 0; kb < C::KB; ++kb)
          tma_load_4d(sb + C::OFF_V + s * C::KVT + kb * C::KVR * 128, &tmV, bar(B_VF + s),
                      kb * 64, j * C::KVR, h, b);
        issued = j + 1;
      }
      if (ab.raised()) {
        // let copies already in flight land before the CTA releases its shared memory
        drain_wait(bar(B_Q), 0);
        for (int j = issued - C::STAGES > 0 ? issued - C::STAGES : 0; j < issued; ++j) {
          const int s = j % C::STAGES, u = j / C::STAGES;
          drain_wait(bar(B_KF + s), u & 1);
          drain_wait(bar(B_VF + s), u & 1);
        }
      }
    }
  } else if (warp == C::W_MMA) {
    // ------------------------------------------------------------------ MMA issuer
    // Warp-uniform: every lane runs the loop and the waits, one elected lane issues.
    constexpr uint32_t idesc_qk = idesc_bf16_f32(BM, C::SK, false, false);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(BM, D, false, true);
    const int total = n_kv * (BN / C::SK);  // scan steps of SK keys
    constexpr int SPL = C::KVR / C::SK;     // scan steps per K/V load unit
    // U of step s = Q K^T over keys [SK s, +SK) into buffer s % NBUF
    auto issue_u = [&](int s) -> bool {
      const int j = s / SPL, hh = s % SPL, st = j % C::STAGES, bf = s % C::NBUF;
      if (hh == 0) {
        if (!mbar_wait_warp(bar(B_KF + st), (j / C::STAGES) & 1, ab)) return false;
        tc_fence_after();
      }
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t koff = (kk >> 2) * (BN * 128) + (kk & 3) * 32;
        const uint32_t kkoff = (kk >> 2) * (C::KVR * 128) + (kk & 3) * 32;
        const uint64_t a = smem_desc_sw128(sb + C::OFF_Q + koff, 16, 1024);
        const uint64_t bd =
            smem_desc_sw128(sb + C::OFF_K + st * C::KVT + hh * C::SK * 128 + kkoff, 16, 1024);
        mma_ss_w(tmem + kSCol + bf * C::SK, a, bd, idesc_qk, kk > 0 ? 1u : 0u);
      }
      mma_commit_w(bar(B_S + bf));  // U ready (and every earlier z update done)
      if (hh == SPL - 1) mma_commit_w(bar(B_KE + st));  // K stage free
      return true;
    };
    bool ok = mbar_wait_warp(bar(B_Q), 0, ab);
    tc_fence_after();
    for (int s0 = 0; ok && s0 < C::NBUF && s0 < total; ++s0) ok = issue_u(s0);
    for (int s = 0; ok && s < total; ++s) {
      const int j = s / SPL, hh = s % SPL, st = j % C::STAGES, bf = s % C::NBUF;
      if (hh == 0 && !(ok = mbar_wait_warp(bar(B_VF + st), (j / C::STAGES) & 1, ab))) break;
      if (!(ok = mbar_wait_warp(bar(B_P + bf), (s / C::NBUF) & 1, ab))) break;
      tc_fence_after();
      // z += P V over the step's SK keys (A = P from TMEM as bf16 pairs in the first
      // SK / 2 columns of the step's buffer; B = V rows, N = d contiguous)
#pragma unroll
      for (int kk = 0; kk < C::SK / 16; ++kk) {
        const uint64_t bd = smem_desc_sw128(
            sb + C::OFF_V + st * C::KVT + (hh * C::SK + kk * 16) * 128, C::KVR * 128, 1024);
        mma_ts_w(tmem + C::OCOL, tmem + kSCol + bf * C::SK + kk * 8, bd, idesc_pv,
                 (s > 0 || kk > 0) ? 1u : 0u);
      }
      mma_commit_w(bar(B_OD + bf));  // z update of step s done
      if (hh == SPL - 1) mma_commit_w(bar(B_VE + st));  // V stage free
      // the next U into the buffer whose P was read above (tcgen05 MMAs run in order)
      if (s + C::NBUF < total && !(ok = issue_u(s + C::NBUF))) break;
    }
    mma_commit_w(bar(B_O));  // z final (or whatever completed before an abort)
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ scan + epilogue
    const int t = threadIdx.x;  // 0..127: row q0 + t, TMEM lane t
    const int r = q0 + t;
    const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
    const float isd = p.inv_sqrt_d;
    const float ch = 0.5f * isd;            // h = U * ch = u / 2
    const float c2k = ch * kLog2e;          // E log2(e) = U * c2k * (1 + tanh(h))
    const float bk = isd * kLog2e;          // bound of E log2 e: max(U, 0) bk (see below)
    // The row's scale m (log2 units): P = 2^(E log2 e - m), l = sum P, z = sum P v, all
    // at the same m.  m is set from the first step's bound of max E, SiLU(u) = u sigma(u)
    // <= max(u, 0) (which exceeds max SiLU by u sigma(-u) <= 0.28, no transcendental), and
    // afterwards every step runs at the scale of the steps before it: its own maximum is
    // taken on the way (not before), and a bound that grew by more than 2^8 raises m once
    // the step's z update has landed (m_next, applied at the next step).  A bound that
    // jumps by more than 2^kStaleLog2 redoes the step at the new scale, so P stays below
    // 2^(kStaleLog2 + 0.28).
    float m = -INFINITY, m_next = -INFINITY;
    float l = 0.f;
    float u_self = 0.f;
    bool ok = true;
    // z (and l) from scale m to mn where `go`, once the z update of step s_done has landed;
    // *scp gets the lane's factor (1 where not `go`)
    auto rescale = [&](bool go, float mn, int s_done, float* scp) -> bool {
      const float sc = go ? ex2_approx(m - mn) : 1.0f;
      if (scp) *scp = sc;
      if (!__any_sync(0xffffffffu, go)) return true;
      if (s_done >= 0) {
        if (!__all_sync(0xffffffffu, mbar_wait(bar(B_OD + s_done % C::NBUF),
                                                (s_done / C::NBUF) & 1, ab)))
          return false;
        tc_fence_after();
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 32) {
          uint32_t z[32];
          tmem_ld32(trow + C::OCOL + c0, z);
          tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < 32; ++c) z[c] = __float_as_uint(__uint_as_float(z[c]) * sc);
          tmem_st16(trow + C::OCOL + c0, z);
          tmem_st16(trow + C::OCOL + c0 + 16, z + 16);
        }
      }
      l *= sc;
      if (go) m = mn;
      return true;
    };
    constexpr int SPT = BN / C::SK;  // scan steps per 128-key tile
    for (int s = 0; s < n_kv * SPT; ++s) {
      const int j = s / SPT, hh = s % SPT, bf = s % C::NBUF;
      ok = __all_sync(0xffffffffu, mbar_wait(bar(B_S + bf), (s / C::NBUF) & 1, ab));
      if (!ok) break;
      tc_fence_after();
      // the larger scale decided at step s - 1, after that step's z update.  Only here:
      // U of step s was issued after the z update of step s - 2 (of step s - 1 with one
      // buffer), so the z-update barrier has completed at least s - 1 phases and its
      // parity wait for phase s - 1 is exact (before the wait above it could still be two
      // phases short and pass at once).
      if (!(ok = rescale(m_next > m, m_next, s - 1, nullptr))) break;
      const uint32_t ucol = trow + kSCol + bf * C::SK;
      // causal: the diagonal tile masks the keys at and after the row (tl, relative to the
      // step's first key); otherwise keys at and past Tk (a ragged last tile) are masked
      const int tl = causal ? t - hh * C::SK : sa.Tk - j * BN - hh * C::SK;
      const bool diag = causal ? (j == qt) : (tl < C::SK);
      float umax;
      float2 rs;
      if constexpr (C::NBUF == 1 || C::SK != HN) {
        // chunks of 32 keys; P of chunk hb written as 16 bf16 pairs to columns 16 hb ..
        // (never ahead of the U columns still to be read) once the chunk's bound is known
        // (a jump in a later chunk also rescales the earlier chunks' P, already in TMEM)
        rs = make_float2(0.f, 0.f);
        umax = -INFINITY;
#pragma unroll
        for (int hb = 0; hb < C::SK / 32; ++hb) {
          uint32_t U[32];
          tmem_ld32(ucol + hb * 32, U);
          tmem_ld_wait();
          const int th = tl - hb * 32;        // the row's index relative to the half
          const bool dg = diag && th < 32;    // some key of the half masked
          if (__any_sync(0xffffffffu, m == -INFINITY)) {
            const float um = dg ? row_max32<true>(U, th, u_self) : row_max32<false>(U, th, u_self);
            if (m == -INFINITY && um != -INFINITY) m = fmaxf(um, 0.f) * bk;
          }
          uint32_t pk[16];
          float mx;
          float2 r = dg ? scan_p32<true>(U, th, ch, c2k, m == -INFINITY ? 0.f : -m, mx, u_self, pk)
                        : scan_p32<false>(U, th, ch, c2k, m == -INFINITY ? 0.f : -m, mx, u_self, pk);
          const float mt = mx == -INFINITY ? -INFINITY : fmaxf(mx, 0.f) * bk;
          const bool jump = mt > m + kStaleLog2;
          if (__any_sync(0xffffffffu, jump)) {
            float sc;
            if (!(ok = rescale(jump, fmaxf(mt, m_next), s - 1, &sc))) break;
            rs = make_float2(rs.x * sc, rs.y * sc);  // the earlier chunks, at the old scale
            if (hb > 0) tmem_st_wait();
            for (int pc = 0; pc < hb; ++pc) {
              uint32_t pa[16];
              tmem_ld16(ucol + pc * 16, pa);
              tmem_ld_wait();
#pragma unroll
              for (int c = 0; c < 16; ++c) {
                const float2 v2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&pa[c]));
                pa[c] = pack_bf16x2(v2.x * sc, v2.y * sc);
              }
              tmem_st16(ucol + pc * 16, pa);
            }
            r = dg ? scan_p32<true>(U, th, ch, c2k, -m, mx, u_self, pk)
                   : scan_p32<false>(U, th, ch, c2k, -m, mx, u_self, pk);
          }
          tmem_st16(ucol + hb * 16, pk);
          rs = __fadd2_rn(rs, r);
          umax = fmaxf(umax, mx);
        }
        if (!ok) break;
      } else {
        static_assert(C::SK == HN, "64-key steps in registers");
        uint32_t U[HN];
        tmem_ld32(ucol, U);
        tmem_ld32(ucol + 32, U + 32);
        tmem_ld_wait();
        // a row that has seen no key yet (z = 0, l = 0) takes this step's bound first
        if (__any_sync(0xffffffffu, m == -INFINITY)) {
          const float um = diag ? row_max<true>(U, tl, u_self) : row_max<false>(U, tl, u_self);
          if (m == -INFINITY && um != -INFINITY) m = fmaxf(um, 0.f) * bk;
        }
        rs = diag ? scan_p<true>(U, tl, ucol, ch, c2k, m == -INFINITY ? 0.f : -m, umax, u_self)
                  : scan_p<false>(U, tl, ucol, ch, c2k, m == -INFINITY ? 0.f : -m, umax, u_self);
        const float mt = umax == -INFINITY ? -INFINITY : fmaxf(umax, 0.f) * bk;
        const bool jump = mt > m + kStaleLog2;  // false while both are -inf
        if (__any_sync(0xffffffffu, jump)) {
          // rare: redo the step at the new scale (z rescaled after step s - 1's update)
          if (!(ok = rescale(jump, fmaxf(mt, m_next), s - 1, nullptr))) break;
          rs = diag ? scan_p<true>(U, tl, ucol, ch, c2k, -m, umax, u_self)
                    : scan_p<false>(U, tl, ucol, ch, c2k, -m, umax, u_self);
        }
      }
      const float mt = umax == -INFINITY ? -INFINITY : fmaxf(umax, 0.f) * bk;
      if (mt > m + kRescaleLog2) m_next = fmaxf(m_next, mt);
      l += rs.x + rs.y;
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(bar(B_P + bf));
    }
    // ---------------------------------------------------------------- epilogue
    // (a scale still pending at the end needs nothing: m, l and z agree)
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar(B_O), 0, ab));
    tc_fence_after();
    if (MODE == 1 && ok) {
      // the Exchange summary of row r: m in natural-log units, l, and z (real columns).
      // The TMEM loads are warp-collective: every lane loads, rows past T store nothing.
      const bool live = r < p.T;
      const long long row = (long long)bh * p.T + r;
      if (live) {
        sa.m[row] = m == -INFINITY ? -INFINITY : m * kLn2;
        sa.l[row] = l;
      }
      float* zr = sa.z + row * p.d;
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32) {
        uint32_t z[32];
        tmem_ld32(trow + C::OCOL + c0, z);
        tmem_ld_wait();
#pragma unroll
        for (int c = 0; c < 32; c += 4)
          if (live && c0 + c < p.d)
            *reinterpret_cast<float4*>(zr + c0 + c) =
                make_float4(__uint_as_float(z[c]), __uint_as_float(z[c + 1]),
                            __uint_as_float(z[c + 2]), __uint_as_float(z[c + 3]));
      }
    } else if (ok) {
      float g = 0.f, inv_l = 0.f, fself = 1.0f;  // F_ii = 1 - g: the Self flow
      float lz;
      const float S = 1.0f / (1.0f + __expf(-(u_self * isd) / p.tau_s));
      if (l > 0.f) {
        const float A = m * kLn2 + __logf(l) - p.lambda * __logf((float)(r + 1));
        g = 1.0f / (1.0f + __expf(S - A));
        fself = 1.0f / (1.0f + __expf(A - S));
        const float hi = fmaxf(S, A), lo = fminf(S, A);
        lz = hi + log1pf(__expf(lo - hi));
        inv_l = 1.0f / l;
      } else {
        lz = S;  // empty history (row 1)
      }
      // v_i from the diagonal tile's V rows, still in shared memory (row t of the stage,
      // 128-byte swizzle); Y staged in the Q tile's space (free: every MMA has completed)
      // and written by one TMA store of 32 rows per warp (rows >= T are clipped).
      // (QUAD: the last two 64-key halves, stages 0 and 1, rows t & 63 of the half t / 64)
      const uint8_t* vrow = C::QUAD
          ? smem + C::OFF_V + (t >> 6) * C::KVT + (t & 63) * 128
          : smem + C::OFF_V + (qt % C::STAGES) * C::KVT + t * 128;
      uint8_t* ystage = smem + C::OFF_Q + warp * (32 * D * 2) + lane * 128;
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32) {
        uint32_t z[32];
        tmem_ld32(trow + C::OCOL + c0, z);
        tmem_ld_wait();
        const int kb = c0 >> 6;  // 64-column block of the tile
#pragma unroll
        for (int c8 = 0; c8 < 32; c8 += 8) {
          const int chunk = ((c0 & 63) + c8) >> 3;  // 16-byte chunk within the 128-byte row
          const uint4 vv = *reinterpret_cast<const uint4*>(vrow + kb * C::KVR * 128 +
                                                           ((chunk ^ (t & 7)) << 4));
          const uint32_t vw[4] = {vv.x, vv.y, vv.z, vv.w};
          uint32_t yw[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 vf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&vw[e]));
            const float z0 = __uint_as_float(z[c8 + 2 * e]) * inv_l;
            const float z1 = __uint_as_float(z[c8 + 2 * e + 1]) * inv_l;
            yw[e] = pack_bf16x2(fmaf(g, z0 - vf.x, vf.x), fmaf(g, z1 - vf.y, vf.y));
          }
          *reinterpret_cast<uint4*>(ystage + kb * (32 * 128) + ((chunk ^ (lane & 7)) << 4)) =
              make_uint4(yw[0], yw[1], yw[2], yw[3]);
        }
      }
      fence_async_smem();
      __syncwarp();
      if (lane == 0) {
        for (int kb = 0; kb < C::KB; ++kb)
          tma_store_4d(&tmO, sb + C::OFF_Q + warp * (32 * D * 2) + kb * (32 * 128), kb * 64,
                       q0 + warp * 32, h, b);
        tma_store_commit();
        tma_store_wait_read_all();  // the staging buffer must outlive the store's reads
      }
      __syncwarp();
      if (r < p.T) {
        p.logz[(long long)bh * p.T + r] = lz;
        if (p.fself) p.fself[(long long)bh * p.T + r] = fself;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == C::W_MMA) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 4-D map over a [B][T][H][d] bf16 tensor: box = 64 columns (128 bytes) x `rows` rows of
// one (h, b), 128-byte swizzle, zero fill outside the tensor.
bool make_tmap_bf16(CUtensorMap* m, const void* base, const Problem& p, int rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {(cuuint64_t)p.d, (cuuint64_t)p.T, (cuuint64_t)p.H, (cuuint64_t)p.B};
  cuuint64_t strides[3] = {(cuuint64_t)p.sT * 2, (cuuint64_t)p.sH * 2, (cuuint64_t)p.sB * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)rows, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// bf16 with d_h a multiple of 8 up to 128: the kernels run at d_pad = 64 or 128, the TMA
// loads filling columns d_h .. d_pad - 1 with zeros (they add nothing to U, z or the
// gradients) and the TMA stores clipping them.
bool supports(relation_dtype dt, int d) {
  return dt == RELATION_BF16 && d >= 8 && d <= 128 && d % 8 == 0;
}

template <int D, int MODE>
static cudaError_t fwd_t(const Problem& p, const StateArgs& sa, cudaStream_t s) {
  // A runtime call first: it makes the primary context current on this thread, which the
  // driver's tensor-map encoder needs.
  const int smem = FwdCfg<D>::SMEM;
  cudaError_t e = cudaFuncSetAttribute(fwd_tc_kernel<D, MODE>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) { note_failure("forward: shared memory attribute"); return e; }
  Problem pk = p;  // the keys' view: their own strides, and count (the state over other keys)
  if (MODE == 1) {
    pk.T = sa.causal ? p.T : sa.Tk;
    pk.sB = sa.k_sB; pk.sT = sa.k_sT; pk.sH = sa.k_sH;
  }
  CUtensorMap mq, mk, mv, mo;
  if (!make_tmap_bf16(&mq, p.q, p, BM) || !make_tmap_bf16(&mk, p.k, pk, FwdCfg<D>::KVR) ||
      !make_tmap_bf16(&mv, p.v, pk, FwdCfg<D>::KVR) ||
      !make_tmap_bf16(&mo, MODE == 0 ? p.out : p.q, p, 32)) {  // (no output tile in MODE 1)
    note_failure("forward: TMA descriptor of Q/K/V/Y");
    return cudaErrorInvalidValue;
  }
  const int n_qt = (p.T + BM - 1) / BM;
  const long long grid = (long long)n_qt * p.B * p.H;
  if (grid > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  int dev = 0, nsm = 148;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    nsm = 148;
  const int groups = head_groups(n_qt, p.B * p.H, FwdCfg<D>::CTAS * nsm);
  fwd_tc_kernel<D, MODE><<<(unsigned)grid, FwdCfg<D>::THREADS, smem, s>>>(mq, mk, mv, mo, p,
                                                                         n_qt, groups, sa);
  if ((e = cudaGetLastError()) != cudaSuccess) note_failure("forward: kernel launch");
  return e;
}

cudaError_t launch_fwd(const Problem& p, cudaStream_t s) {
  if (!supports(p.dtype, p.d)) return cudaErrorInvalidValue;
  StateArgs none{};
  none.causal = 1;
  return p.d <= 64 ? fwd_t<64, 0>(p, none, s) : fwd_t<128, 0>(p, none, s);
}

cudaError_t launch_fwd_state(const Problem& p, const StateArgs& sa, cudaStream_t s) {
  if (!supports(p.dtype, p.d) || !sa.m || !sa.l || !sa.z || (!sa.causal && sa.Tk < 1))
    return cudaErrorInvalidValue;
  return p.d <= 64 ? fwd_t<64, 1>(p, sa, s) : fwd_t<128, 1>(p, sa, s);
}

}  // namespace tc
}  // namespace rel
