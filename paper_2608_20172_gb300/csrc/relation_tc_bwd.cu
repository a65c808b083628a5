// relation_tc_bwd.cu -- tcgen05 / TMA / TMEM backward of FlashRelation (bf16, d_h 64/128).
//
// Gradient of the causal Relation row softmax (App. A.1.7, generic form).  For every
// pair j <= i of one head, with F the flow and G = dL/dY:
//   dR_ij = F_ij (dO_i . v_j - D_i),   D_i = dO_i . Y_i
//   dS_ij = dR_ij SiLU'(u_ij)                    (Exchange, j < i)
//   dS_ii = dR_ii S_i (1 - S_i) / tau_S          (Self, j = i; S_i = sigmoid(u_ii / tau_S))
//   dV_j += F_ij dO_i,  dK_j += dS_ij q_i / sqrt(d),  dQ_i += dS_ij k_j / sqrt(d)
// with F_ij = exp(E_ij - lambda log i - logZ_i) (j < i) and F_ii = exp(S_i - logZ_i).
// The Self entries (j = i) are computed per row in fp32 by the row pass; the tile kernel
// computes the Exchange pairs (j < i) and places the Self values on the diagonal of its
// diagonal tile, so that its dV, dK and dQ products include them.
//
// Three launches: a row pass (D_i, the Self entries and their dlambda terms, the tile
// kernel's per-query scalars, zeroed fp32 dQ accumulator), the tile kernel, and a
// finalisation (dQ to bf16, dlambda reduction).
//
// Tile kernel: a unit is 128 keys of one head, visiting query tiles from the diagonal to
// the end of the sequence; d_h = 64 runs one persistent CTA per SM over the units (K/V
// double-buffered, the next unit's first steps issued before the current unit's last dQ),
// d_h = 128 one CTA per unit.  Keys sit on TMEM lanes.  Per step of 64 query columns:
//   MMA  U^T = K Q^T,  dP^T = V dO^T                          (TMEM, fp32)
//   elementwise (thread = key): P = F in bf16 back into TMEM, dS' = 2 dS in bf16 into
//        128-byte-swizzled shared memory, and the Exchange part of dlambda
//   MMA  dV += P^T dO (P read from TMEM),  dK += dS'^T Q
// Two TMEM buffers of U^T / dP^T: the MMAs of one buffer (dV, dK of the last step, U^T /
// dP^T of the next) overlap the elementwise work on the other; every elementwise
// warpgroup works on every step (d_h = 64: four warpgroups of 16 query columns, d_h = 128:
// two of 32).  dQ goes to an fp32 accumulator through TMA reduce-add,
// staged by the four dQ warps (after the elementwise warps):
//   d_h = 64 : dQ_t = dS' K once per 128-query tile, in TMEM columns of its own.
//   d_h = 128: dQ^T = K^T dS'^T once per step (d on TMEM lanes), written into the step's
//              dP^T columns after dK has read dS' (TMEM is full otherwise); the next U^T
//              of the buffer is issued after it, the next dP^T after its read-out.
// A tcgen05.mma costs at least ~46 cycles whatever its N (measured on GB300: N = 32, 64,
// 128 run at 35%, 66%, 99% of the per-SM peak), so the steps keep N >= 64.
// dlambda = sum_i log i (1 - F_ii) dR_ii - sum_{j<i} log i F_ii dR_ij: the row pass sums
// the first part per block, the tile kernel the second per CTA.  In exact arithmetic it
// equals sum_i log i dR_ii; this weighting cancels the rounding error of D_i (see
// aux_kernels.cu).
#include <cudaTypedefs.h>
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rel {
namespace tc {

bool make_tmap_bf16(CUtensorMap* m, const void* base, const Problem& p, int rows);

namespace bwd {

constexpr int BK = 128;        // keys per CTA
constexpr int BT = 128;        // queries per TMA tile
// Warps: 4 NWG elementwise (NWG warpgroups, Cfg), then 4 dQ, 1 TMA, 1 MMA.
constexpr int kTmemCols = 512;


template <int D>
struct Cfg {
  static constexpr int KB = D / 64;
  static constexpr int KVT = 128 * D * 2;  // one K or V tile
  // Q / dO staging and the dQ product:
  //   d_h = 64 : per 128-query tile (two stages); dQ_t = dS' K once per tile into its own
  //              TMEM columns.
  //   d_h = 128: per 64-query step (three stages); dQ^T = K^T dS'^T once per step into the
  //              step's own dP^T columns, after dK has read dS' out of them.
  static constexpr bool HALF = D == 128;
  static constexpr int NBUF = 2;               // U^T / dP^T TMEM buffers
  static constexpr int QW = 64;                // query columns per step
  static constexpr int SPT = BT / QW;          // steps per query tile
  static constexpr int QROWS = HALF ? QW : BT; // query rows per Q / dO stage
  static constexpr int QSZ = QROWS * D * 2;    // bytes of one Q (or dO) stage (16 KB)
  static constexpr int KBQ = QROWS * 128;      // stride of the 64-column blocks of a stage
  static constexpr int NQS = HALF ? 3 : 2;     // Q / dO stages
  static constexpr int SW = QROWS;             // per-query scalars of a stage: array stride
  static constexpr int STB = 3 * SW * 4;       // bytes of one stage's scalars
  static constexpr int DSZ = HALF ? 16384 : 32768;  // one dS' buffer (per step / per tile)
  static constexpr int DQSLOTS = 1;                 // 4 KB staging slot per dQ warp
  // K / V buffers: d_h = 64 runs persistent CTAs and loads the next unit's K and V while
  // the current unit runs; d_h = 128 takes one unit per CTA.
  static constexpr int NKV = HALF ? 1 : 2;
  static constexpr int OFF_KV = 0;                  // buffer k: K at + 2 KVT k, V after it
  static constexpr int OFF_Q = OFF_KV + NKV * 2 * KVT;
  static constexpr int OFF_DO = OFF_Q + NQS * QSZ;
  static constexpr int OFF_DS = OFF_DO + NQS * QSZ;
  static constexpr int OFF_DQS = OFF_DS + 2 * DSZ;
  static constexpr int OFF_STAT = OFF_DQS + 4 * DQSLOTS * 4096;
  static constexpr int OFF_RED = OFF_STAT + NQS * STB;
  static constexpr int OFF_BAR = OFF_RED + 64;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  // Elementwise warpgroups: four at d_h = 64 (each takes 16 query columns of a step: more
  // warps per SMSP hide the latency of the step's loads), two at d_h = 128 (32 columns
  // each, in two halves of 16; the MMAs bound that path and a larger CTA spills).
  static constexpr int NWG = D == 64 ? 4 : 2;
  static constexpr int CW = QW / NWG;          // query columns per warpgroup and step
  static constexpr int EW_THREADS = 128 * NWG;
  static constexpr int W_DQ = 4 * NWG, W_TMA = W_DQ + 4, W_MMA = W_DQ + 5;
  static constexpr int THREADS = 32 * (W_MMA + 1);
  static constexpr int COL_DK = NBUF * 2 * QW;  // 256
  static constexpr int COL_DV = COL_DK + D;     // 320 / 384
  static constexpr int COL_DQ = 384;            // d_h = 64 only
  // d_h = 64: the unit's K and V tiles also in TMEM (A operands of U^T = K Q^T and
  // dP^T = V dO^T, which then read only Q / dO from shared memory: an SS MMA at N = 64
  // reads 6 KB of operands in 48 cycles of shared-memory bandwidth against 32 of math)
  static constexpr int COL_KT = 448, COL_VT = 480;
  static_assert(HALF || COL_VT + D / 2 <= 512, "TMEM");
  __host__ __device__ static constexpr int col_u(int b) { return b * 2 * QW; }
  __host__ __device__ static constexpr int col_g(int b) { return b * 2 * QW + QW; }
  // Q / dO stage unit of a step: the step itself (d_h = 128) or its query tile
  __host__ __device__ static constexpr int unit_of(int s) { return HALF ? s : s / SPT; }
};
static_assert(Cfg<64>::SMEM <= 232448 && Cfg<128>::SMEM <= 232448, "shared memory");

enum : int {
  B_KV = 0, B_QF = 1, B_QE = 4, B_S = 7, B_P = 9, B_DQF = 11, B_DQE = 13, B_ACC = 15,
  B_KVE = 16, B_STG = 18, B_KV1 = 19  // B_KVE + k: K / V buffer k free; B_KV1: buffer 1 full
};
__device__ __forceinline__ int kv_full(int k) { return k == 0 ? B_KV : B_KV1; }

__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > 20ull * 1000ull * 1000ull) return;
  }
}

__device__ __forceinline__ void tma_reduce_add_2d(const CUtensorMap* m, uint32_t src, int c0,
                                                  int c1) {
  asm volatile(
      "cp.reduce.async.bulk.tensor.2d.global.shared::cta.add.tile.bulk_group [%0, {%2, %3}], [%1];"
      ::"l"(reinterpret_cast<uint64_t>(m)), "r"(src), "r"(c0), "r"(c1)
      : "memory");
}
// 1-D bulk copy global -> shared completing on an mbarrier (16-byte aligned, size % 16 == 0)
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void bulk_wait_read_0() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}

// Per-thread constants of the elementwise step.
struct EwConst {
  float ch;   // u / 2 = U ch       (U = raw q . k, u = U / sqrt(d))
  float c2k;  // E log2 e = U c2k (1 + tanh(u / 2))
};

// Elementwise work on 32 query columns of one key row (this thread's key t), Exchange
// entries only.  st points at the chunk's first query in the stage's per-query scalars,
// three arrays of stride SW: [0] c2 = (-lambda log i - logZ_i) log2 e, [SW] -D_i,
// [2 SW] -log i F_ii.  qt0 is the tile-local index of the chunk's first query.
// Produces P = F_ij and dS' = 2 dS_ij as bf16 pairs and accumulates the dlambda terms:
//   P = 2^(U c2k (1 + t) + c2),  t = tanh(u/2),
//   2 SiLU'(u) = a (1 + h (1 - t)) with a = 1 + t, h = u / 2.
// On the diagonal tile (DIAG) the entries with query <= key get c2 = -inf, so P, dS' and
// their dlambda terms are exactly zero; the Self entry (query == key) then takes the
// row pass's values, P = F_tt and dS' = 2 dS_tt (self2 = {F_tt, dS_tt}), so that the
// dV, dK and dQ products include it (its dlambda term is the row pass's).
template <bool DIAG, int SW, int N>
__device__ __forceinline__ void ew_chunk(const uint32_t (&U)[N], const uint32_t (&G)[N],
                                         const float* st, int qt0, int t, const EwConst& k,
                                         float2 self2, uint32_t (&pk)[N / 2],
                                         uint32_t (&dk)[N / 2], float2& dl2) {
  const float2 ch2 = make_float2(k.ch, k.ch), c2k2 = make_float2(k.c2k, k.c2k);
  const float2 one2 = make_float2(1.f, 1.f);
#pragma unroll
  for (int c = 0; c < N; c += 4) {
    float4 c2v = *reinterpret_cast<const float4*>(st + c);
    const float4 ndv = *reinterpret_cast<const float4*>(st + SW + c);
    const float4 nwv = *reinterpret_cast<const float4*>(st + 2 * SW + c);
    if (DIAG) {  // keep query > key
      const int q = qt0 + c;
      c2v.x = q > t ? c2v.x : -INFINITY;
      c2v.y = q + 1 > t ? c2v.y : -INFINITY;
      c2v.z = q + 2 > t ? c2v.z : -INFINITY;
      c2v.w = q + 3 > t ? c2v.w : -INFINITY;
    }
#pragma unroll
    for (int e = 0; e < 4; e += 2) {
      const float2 x = make_float2(__uint_as_float(U[c + e]), __uint_as_float(U[c + e + 1]));
      const float2 g = make_float2(__uint_as_float(G[c + e]), __uint_as_float(G[c + e + 1]));
      const float2 c2 = e == 0 ? make_float2(c2v.x, c2v.y) : make_float2(c2v.z, c2v.w);
      const float2 nd = e == 0 ? make_float2(ndv.x, ndv.y) : make_float2(ndv.z, ndv.w);
      const float2 nw = e == 0 ? make_float2(nwv.x, nwv.y) : make_float2(nwv.z, nwv.w);
      const float2 h = __fmul2_rn(x, ch2);
      const float2 th = make_float2(tanh_approx(h.x), tanh_approx(h.y));
      const float2 a = __fadd2_rn(th, one2);
      const float2 w = __fmul2_rn(a, c2k2);
      const float2 ex = __ffma2_rn(x, w, c2);
      const float2 P = make_float2(ex2_approx(ex.x), ex2_approx(ex.y));
      const float2 dR = __fmul2_rn(P, __fadd2_rn(g, nd));
      const float2 b = __ffma2_rn(make_float2(-h.x, -h.y), th, h);  // h (1 - t)
      const float2 sp = __ffma2_rn(a, b, a);                        // 2 SiLU'(u)
      float2 dS = __fmul2_rn(dR, sp);
      dl2 = __ffma2_rn(nw, dR, dl2);
      float2 Pv = P;
      if (DIAG) {
        const int q = qt0 + c + e;
        if (q == t) { Pv.x = self2.x; dS.x = 2.0f * self2.y; }
        if (q + 1 == t) { Pv.y = self2.x; dS.y = 2.0f * self2.y; }
      }
      pk[(c + e) >> 1] = pack_bf16x2(Pv.x, Pv.y);
      dk[(c + e) >> 1] = pack_bf16x2(dS.x, dS.y);
    }
  }
}

template <int D>
__global__ void __launch_bounds__(Cfg<D>::THREADS, 1)
    bwd_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmG,
                  const __grid_constant__ CUtensorMap tmDQ, const __grid_constant__ CUtensorMap tmDK,
                  const __grid_constant__ CUtensorMap tmDV, Problem p, BwdWorkspace ws, int n_t,
                  int t_pad, int n_groups) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sb = smem_u32(smem);
  auto bar = [&](int i) -> uint32_t { return sb + C::OFF_BAR + 8u * (uint32_t)i; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_BAR + 192);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_BAR + 200);
  float* red = reinterpret_cast<float*>(smem + C::OFF_RED);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int BH = p.B * p.H;
  const int n_work = n_t * BH;  // work units (key tile, head), most query tiles first, heads
                                // in groups (grouped_unit)
  // A unit: keys kt * 128 .. of head bh, query tiles kt .. n_t - 1.  Round r of the grid
  // takes units r G .. r G + G - 1 (G = gridDim.x), CTA c the unit r G + c in even rounds
  // and r G + G - 1 - c in odd ones: the units come heaviest first, so the zigzag evens
  // out the CTAs' work.  Every role walks the same sequence and keeps running counts
  // (units, steps, Q / dO stage loads, query tiles) from which the barrier phases follow.
  // d_h = 128 takes one unit per CTA (the launch gives one CTA per unit): its loops over
  // units end after the first at compile time.
  auto unit_at = [&](int r) -> int {
    if (C::HALF) return r == 0 ? (int)blockIdx.x : n_work;
    const int c = (r & 1) ? (int)(gridDim.x - 1 - blockIdx.x) : (int)blockIdx.x;
    return r * (int)gridDim.x + c;
  };
  struct Unit {
    int kt, bh, b, h, k0, n_i, total, n_units;
  };
  auto unit = [&](int w) {
    Unit u;
    grouped_unit(w, n_t, BH, n_groups, u.kt, u.bh);
    u.b = u.bh / p.H;
    u.h = u.bh % p.H;
    u.k0 = u.kt * BK;
    u.n_i = n_t - u.kt;
    u.total = u.n_i * C::SPT;
    u.n_units = C::HALF ? u.total : u.n_i;
    return u;
  };

  if (threadIdx.x == 0) {
    for (int k = 0; k < C::NKV; ++k) {
      mbar_init(bar(kv_full(k)), 1);
      mbar_init(bar(B_KVE + k), 1);
    }
    for (int s = 0; s < C::NQS; ++s) {
      mbar_init(bar(B_QF + s), 1);
      mbar_init(bar(B_QE + s), 1);
    }
    for (int s = 0; s < C::NBUF; ++s) {
      mbar_init(bar(B_S + s), 1);
      mbar_init(bar(B_P + s), C::EW_THREADS);  // every elementwise warpgroup
      mbar_init(bar(B_DQF + s), 1);
      mbar_init(bar(B_DQE + s), 128);
    }
    mbar_init(bar(B_ACC), 1);
    mbar_init(bar(B_STG), C::EW_THREADS);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == C::W_MMA) tmem_alloc(smem_u32(tmem_slot), kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const Abort ab{abort_flag, p.dev_status};

  if (warp == C::W_TMA) {
    // ------------------------------------------------------ TMA + per-query scalars
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmG);
      tma_prefetch_desc(&tmDK);
      tma_prefetch_desc(&tmDV);
      bool ok = true;
      int ul = 0, gq0 = 0, kv_issued = 0, q_issued = 0;
      // Q / dO stage load g (global count) for local unit u of U
      auto load_q = [&](const Unit& U, int u) -> bool {
        const int g = gq0 + u, s = g % C::NQS, r = g / C::NQS;
        if (r > 0 && !mbar_wait(bar(B_QE + s), (r - 1) & 1, ab)) return false;
        const int tile = C::HALF ? u / C::SPT : u;
        const int qoff = C::HALF ? (u % C::SPT) * C::QW : 0;
        const int qi0 = (U.kt + tile) * BT + qoff;
        mbar_arrive_expect_tx(bar(B_QF + s), 2 * C::QSZ + C::STB);
        for (int kb = 0; kb < C::KB; ++kb) {
          tma_load_4d(sb + C::OFF_Q + s * C::QSZ + kb * C::KBQ, &tmQ, bar(B_QF + s), kb * 64,
                      qi0, U.h, U.b);
          tma_load_4d(sb + C::OFF_DO + s * C::QSZ + kb * C::KBQ, &tmG, bar(B_QF + s), kb * 64,
                      qi0, U.h, U.b);
        }
        const float* src = ws.stats + ((long long)U.bh * n_t + U.kt + tile) * 3 * BT + qoff;
        if (C::HALF) {
          for (int a = 0; a < 3; ++a)
            bulk_load(sb + C::OFF_STAT + s * C::STB + a * C::SW * 4, src + a * BT, C::SW * 4,
                      bar(B_QF + s));
        } else {
          bulk_load(sb + C::OFF_STAT + s * C::STB, src, C::STB, bar(B_QF + s));
        }
        q_issued = g + 1;
        return true;
      };
      for (int w; ok && (w = unit_at(ul)) < n_work; ++ul) {
        const Unit U = unit(w);
        // K / V into buffer ul % NKV once the last MMA of the unit that used it before
        // (unit ul - NKV) has completed; with two buffers this load overlaps the previous
        // unit's work
        const int kvb = ul % C::NKV;
        const uint32_t kvs = sb + C::OFF_KV + kvb * 2 * C::KVT;
        if (ul >= C::NKV && !(ok = mbar_wait(bar(B_KVE + kvb), ((ul - C::NKV) / C::NKV) & 1, ab)))
          break;
        mbar_arrive_expect_tx(bar(kv_full(kvb)), 2 * C::KVT);
        for (int kb = 0; kb < C::KB; ++kb) {
          tma_load_4d(kvs + kb * 16384, &tmK, bar(kv_full(kvb)), kb * 64, U.k0, U.h, U.b);
          tma_load_4d(kvs + C::KVT + kb * 16384, &tmV, bar(kv_full(kvb)), kb * 64, U.k0, U.h, U.b);
        }
        ++kv_issued;
        for (int u = 0; ok && u < U.n_units; ++u) ok = load_q(U, u);
        gq0 += U.n_units;
      }
      if (ab.raised()) {
        // let copies already in flight land before the CTA releases its shared memory
        for (int k = kv_issued - C::NKV > 0 ? kv_issued - C::NKV : 0; k < kv_issued; ++k)
          drain_wait(bar(kv_full(k % C::NKV)), (k / C::NKV) & 1);
        for (int g = q_issued - C::NQS > 0 ? q_issued - C::NQS : 0; g < q_issued; ++g)
          drain_wait(bar(B_QF + g % C::NQS), (g / C::NQS) & 1);
      }
    }
  } else if (warp == C::W_MMA) {
    // ------------------------------------------------------ MMA issuer
    // Warp-uniform: every lane runs the loop and the waits, one elected lane issues.
    constexpr uint32_t id_s = idesc_bf16_f32(128, C::QW, false, false);  // U^T, dP^T
    constexpr uint32_t id_acc = idesc_bf16_f32(128, D, false, true);     // dV, dK
    constexpr uint32_t id_dq = C::HALF ? idesc_bf16_f32(128, C::QW, true, true)  // dQ^T
                                       : idesc_bf16_f32(128, D, true, true);     // dQ
    bool ok = true;
    bool acc_done = false;  // B_ACC of the current unit committed
    // A unit's running offsets (steps, Q / dO stage loads) and its K / V tiles
    struct Ctx {
      int gs0, gq0;
      uint32_t ks, vs;
    };
    auto ctx_of = [&](int ul_, int gs0_, int gq0_) {
      const uint32_t k = sb + C::OFF_KV + (ul_ % C::NKV) * 2 * C::KVT;
      return Ctx{gs0_, gq0_, k, k + C::KVT};
    };
    // U^T of step s into buffer (gs0 + s) % NBUF (waits for its Q / dO stage)
    auto issue_u = [&](const Ctx& x, int s) -> bool {
      const int g = x.gq0 + C::unit_of(s), st = g % C::NQS, bb = (x.gs0 + s) % C::NBUF;
      const int hh = s % C::SPT;
      if (C::HALF || hh == 0) {
        if (!mbar_wait_warp(bar(B_QF + st), (g / C::NQS) & 1, ab)) return false;
        tc_fence_after();
      }
      const uint32_t rows = C::HALF ? 0u : (uint32_t)(hh * C::QW * 128);  // the step's rows
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t kof = (kk >> 2) * 16384 + (kk & 3) * 32;
        const uint32_t qof = (kk >> 2) * C::KBQ + (kk & 3) * 32;
        const uint64_t bq = smem_desc_sw128(sb + C::OFF_Q + st * C::QSZ + rows + qof, 16, 1024);
        if (C::HALF)
          mma_ss_w(tmem + C::col_u(bb), smem_desc_sw128(x.ks + kof, 16, 1024), bq, id_s,
                   kk > 0 ? 1u : 0u);
        else
          mma_ts_w(tmem + C::col_u(bb), tmem + C::COL_KT + kk * 8, bq, id_s, kk > 0 ? 1u : 0u);
      }
      return true;
    };
    // dP^T of step s (after issue_u(s)), then the step's S barrier
    auto issue_dp = [&](const Ctx& x, int s) {
      const int st = (x.gq0 + C::unit_of(s)) % C::NQS, bb = (x.gs0 + s) % C::NBUF;
      const int hh = s % C::SPT;
      const uint32_t rows = C::HALF ? 0u : (uint32_t)(hh * C::QW * 128);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t kof = (kk >> 2) * 16384 + (kk & 3) * 32;
        const uint32_t qof = (kk >> 2) * C::KBQ + (kk & 3) * 32;
        const uint64_t bg = smem_desc_sw128(sb + C::OFF_DO + st * C::QSZ + rows + qof, 16, 1024);
        if (C::HALF)
          mma_ss_w(tmem + C::col_g(bb), smem_desc_sw128(x.vs + kof, 16, 1024), bg, id_s,
                   kk > 0 ? 1u : 0u);
        else
          mma_ts_w(tmem + C::col_g(bb), tmem + C::COL_VT + kk * 8, bg, id_s, kk > 0 ? 1u : 0u);
      }
      mma_commit_w(bar(B_S + bb));
    };
    // d_h = 64: the unit's K and V tiles into TMEM (in order after every earlier MMA, so the
    // previous unit's products have read the old ones)
    auto load_kv_tmem = [&](const Ctx& x) {
      if (!C::HALF) {
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          tmem_cp_w(tmem + C::COL_KT + kk * 8, smem_desc_sw128(x.ks + kk * 32, 16, 1024));
          tmem_cp_w(tmem + C::COL_VT + kk * 8, smem_desc_sw128(x.vs + kk * 32, 16, 1024));
        }
      }
    };
    int ul = 0, gs0 = 0, gq0 = 0, gt0 = 0;
    int pre = 0;  // steps of the current unit issued ahead by the previous unit
    for (int w; ok && (w = unit_at(ul)) < n_work; ++ul) {
      const Unit U = unit(w);
      const int total = U.total;
      acc_done = false;
      const int kvb = ul % C::NKV;
      const Ctx x = ctx_of(ul, gs0, gq0);
      const uint32_t ks = x.ks;
      if (pre == 0) {
        if (!(ok = mbar_wait_warp(bar(kv_full(kvb)), (ul / C::NKV) & 1, ab))) break;
        tc_fence_after();
        load_kv_tmem(x);
      }
      // d_h = 64: U^T / dP^T of step sn may be issued once its buffer is free (step
      // sn - NBUF done) and once the GEMM that releases the Q/dO stage it loads into has
      // been issued: waiting for that stage's load earlier would deadlock.
      int sn = pre, units_done = 0;
      pre = 0;
      while (ok && sn < total && sn < C::NBUF) {
        ok = issue_u(x, sn);
        if (ok) issue_dp(x, sn);
        ++sn;
      }
      for (int s = 0; ok && s < total; ++s) {
        const int t = s / C::SPT, hh = s % C::SPT, g = gs0 + s, bb = g % C::NBUF;
        const int st = (gq0 + C::unit_of(s)) % C::NQS;
        if (!(ok = mbar_wait_warp(bar(B_P + bb), (g / C::NBUF) & 1, ab))) break;
        tc_fence_after();
        // dV += P^T dO and dK += dS'^T Q with the A operands in TMEM: every 32-query chunk
        // keeps its 16 packed columns of P (dS') at the start of its own U^T (dP^T)
        // columns.  The first step of a unit starts the sums afresh; the epilogue has
        // read the previous unit's sums before its warps finished this step (B_P).
        const uint32_t pcol = C::col_u(bb), dcol = C::col_g(bb);
        const uint32_t rows = C::HALF ? 0u : (uint32_t)(hh * C::QW * 128);
#pragma unroll
        for (int kk = 0; kk < C::QW / 16; ++kk) {
          constexpr int H = C::CW / 16;  // 16-query chunks per warpgroup
          const uint32_t acol = (kk / H) * C::CW + (kk % H) * 8;
          mma_ts_w(tmem + C::COL_DV, tmem + pcol + acol,
                   smem_desc_sw128(sb + C::OFF_DO + st * C::QSZ + rows + kk * 2048, C::KBQ, 1024),
                   id_acc, (s > 0 || kk > 0) ? 1u : 0u);
        }
#pragma unroll
        for (int kk = 0; kk < C::QW / 16; ++kk) {
          constexpr int H = C::CW / 16;
          const uint32_t acol = (kk / H) * C::CW + (kk % H) * 8;
          mma_ts_w(tmem + C::COL_DK, tmem + dcol + acol,
                   smem_desc_sw128(sb + C::OFF_Q + st * C::QSZ + rows + kk * 2048, C::KBQ, 1024),
                   id_acc, (s > 0 || kk > 0) ? 1u : 0u);
        }
        if (s == total - 1) {  // dK and dV are final: the epilogue need not wait for dQ
          mma_commit_w(bar(B_ACC));
          acc_done = true;
          // d_h = 64: the next unit's first steps go ahead of this unit's last dQ (their
          // buffers were read by the dV / dK just issued; its K / V came in beforehand)
          const int wn = C::HALF ? n_work : unit_at(ul + 1);
          if (wn < n_work) {
            const Unit N = unit(wn);
            if (!(ok = mbar_wait_warp(bar(kv_full((ul + 1) % C::NKV)), ((ul + 1) / C::NKV) & 1, ab)))
              break;
            const Ctx xn = ctx_of(ul + 1, gs0 + total, gq0 + U.n_units);
            tc_fence_after();
            load_kv_tmem(xn);
            while (ok && pre < N.total && pre < C::NBUF) {
              ok = issue_u(xn, pre);
              if (ok) issue_dp(xn, pre);
              ++pre;
            }
            if (!ok) break;
          }
        }
        if (C::HALF) {
          mma_commit_w(bar(B_QE + st));  // the step's Q / dO rows are no longer needed
          // Buffer bb next holds step s + 2.  Issue order (executed in order): dQ^T of
          // step s over dS' in the dP^T columns, which dK has read; U^T of step s + 2
          // over P, which dV has read; dP^T of step s + 2 once dQ^T has been read out.
          // dQ^T = K^T dS'^T (A = K tile, d-major; B = the step's dS', query-major)
          const uint32_t dsb = sb + C::OFF_DS + (g & 1) * C::DSZ;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            mma_ss_w(tmem + C::col_g(bb), smem_desc_sw128(ks + kk * 2048, 16384, 1024),
                     smem_desc_sw128(dsb + kk * 2048, 16384, 1024), id_dq, kk > 0 ? 1u : 0u);
          mma_commit_w(bar(B_DQF + bb));
          const int s2 = s + C::NBUF;
          if (s2 < total && !(ok = issue_u(x, s2))) break;
          if (s2 < total) {
            if (!(ok = mbar_wait_warp(bar(B_DQE + bb), (g / C::NBUF) & 1, ab))) break;
            tc_fence_after();
            issue_dp(x, s2);
          }
          continue;
        }
        if (hh == C::SPT - 1) {
          const int gt = gt0 + t;
          if (gt > 0) {  // dQ of the previous query tile has been read out of TMEM
            if (!(ok = mbar_wait_warp(bar(B_DQE), (gt - 1) & 1, ab))) break;
            tc_fence_after();
          }
          // dQ_t = dS' K   (A = dS', queries x keys, M-major; B = K tile, N-major)
          const uint32_t ds_base = sb + C::OFF_DS + (gt & 1) * C::DSZ;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            mma_ss_w(tmem + C::COL_DQ, smem_desc_sw128(ds_base + kk * 2048, 16384, 1024),
                     smem_desc_sw128(ks + kk * 2048, 16384, 1024), id_dq,
                     kk > 0 ? 1u : 0u);
          mma_commit_w(bar(B_DQF));
          mma_commit_w(bar(B_QE + st));
          ++units_done;
        }
        while (ok && sn < total && sn <= s + C::NBUF &&
               C::unit_of(sn) - C::NQS < units_done) {
          ok = issue_u(x, sn);
          if (ok) issue_dp(x, sn);
          ++sn;
        }
      }
      if (!ok) break;
      mma_commit_w(bar(B_KVE + kvb));  // every MMA of the unit (K / V buffer free) done
      gs0 += total;
      gq0 += U.n_units;
      gt0 += U.n_i;
    }
    if (!acc_done) mma_commit_w(bar(B_ACC));  // after an abort: whatever completed
    __syncwarp();
  } else if (warp >= C::W_DQ) {
    // ------------------------------------------------------ dQ -> fp32 accumulator
    const int quad = warp & 3;
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const uint32_t stage0 = sb + C::OFF_DQS + quad * C::DQSLOTS * 4096;
    uint8_t* stage0p = smem + C::OFF_DQS + quad * C::DQSLOTS * 4096;
    bool ok = true;
    int gs0 = 0, gt0 = 0, chunk = 0;
    for (int r = 0, w; ok && (w = unit_at(r)) < n_work; ++r) {
      const Unit U = unit(w);
      if (C::HALF) {
        // TMEM lanes are d indices here: this warp holds d = 32 quad .. 32 quad + 31 of the
        // step's 64 queries and writes them as 32-query x 32-d boxes, transposed.
        for (int s = 0; s < U.total; ++s) {
          const int g = gs0 + s, bb = g % C::NBUF;
          ok = __all_sync(0xffffffffu, mbar_wait(bar(B_DQF + bb), (g / C::NBUF) & 1, ab));
          if (!ok) break;
          tc_fence_after();
          uint32_t z[64];
          tmem_ld32(trow + C::col_g(bb), z);
          tmem_ld32(trow + C::col_g(bb) + 32, z + 32);
          tmem_ld_wait();
          tc_fence_before();
          mbar_arrive(bar(B_DQE + bb));  // the buffer may take the next dP^T
          const int row0 = U.bh * t_pad + (U.kt + s / C::SPT) * BT + (s % C::SPT) * C::QW;
          const uint32_t sw = (uint32_t)(lane & 3) << 2;
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            if (lane == 0) bulk_wait_read_0();  // the slot's previous reduce has read it
            __syncwarp();
#pragma unroll
            for (int q = 0; q < 32; ++q)
              *reinterpret_cast<uint32_t*>(stage0p + q * 128 + (((lane >> 2) ^ (q & 7)) << 4) +
                                           sw) = z[c * 32 + q];
            fence_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_reduce_add_2d(&tmDQ, stage0, quad * 32, row0 + c * 32);
              tma_store_commit();
            }
          }
        }
      } else {
        for (int i = 0; i < U.n_i; ++i) {
          const int gt = gt0 + i;
          ok = __all_sync(0xffffffffu, mbar_wait(bar(B_DQF), gt & 1, ab));
          if (!ok) break;
          tc_fence_after();
          const int row0 = U.bh * t_pad + (U.kt + i) * BT + quad * 32;
#pragma unroll
          for (int c64 = 0; c64 < D; c64 += 64) {
            uint32_t z[64];
            tmem_ld32(trow + C::COL_DQ + c64, z);
            tmem_ld32(trow + C::COL_DQ + c64 + 32, z + 32);
            tmem_ld_wait();
            if (c64 + 64 == D) {
              tc_fence_before();
              mbar_arrive(bar(B_DQE));  // TMEM columns free for the next dQ
            }
#pragma unroll
            for (int c0 = 0; c0 < 64; c0 += 32, ++chunk) {
              const int slot = chunk % C::DQSLOTS;
              if (lane == 0) bulk_wait_read_0();  // the slot's previous reduce has read it
              __syncwarp();
              uint8_t* row = stage0p + slot * 4096 + lane * 128;
#pragma unroll
              for (int k = 0; k < 8; ++k)
                *reinterpret_cast<uint4*>(row + ((k ^ (lane & 7)) << 4)) =
                    make_uint4(z[c0 + 4 * k], z[c0 + 4 * k + 1], z[c0 + 4 * k + 2], z[c0 + 4 * k + 3]);
              fence_async_smem();
              __syncwarp();
              if (lane == 0) {
                tma_reduce_add_2d(&tmDQ, stage0 + slot * 4096, c64 + c0, row0);
                tma_store_commit();
              }
            }
          }
        }
      }
      gs0 += U.total;
      gt0 += U.n_i;
    }
    if (lane == 0) tma_store_wait_read_all();  // the staging reads; the adds finish with the kernel
  } else {
    // ------------------------------------------------------ elementwise + epilogue
    // Both warpgroups work on every step: warpgroup wg takes its 32 query columns.
    const int wg = warp >> 2;                  // 0 or 1
    const int t = (warp & 3) * 32 + lane;      // key k0 + t, TMEM lane t
    const int wq = warp & 3;
    const uint32_t trow = tmem + ((uint32_t)(wq * 32) << 16);
    const float isd = p.inv_sqrt_d;
    EwConst kc;
    kc.ch = 0.5f * isd;
    kc.c2k = kc.ch * kLog2e;
    float2 dl2 = make_float2(0.f, 0.f);
    bool ok = true;
    int ul = 0, gs0 = 0, gq0 = 0, gt0 = 0;
    for (int w; ok && (w = unit_at(ul)) < n_work; ++ul) {
      const Unit U = unit(w);
      // The Self entry of this thread's key (row pass), placed on the diagonal tile's
      // diagonal; keys past T read a clamped row (their products are never stored).
      const long long self_row = (long long)U.bh * p.T + min(U.k0 + t, p.T - 1);
      const float2 self2 = make_float2(ws.F_self[self_row], ws.dS_self[self_row]);
      for (int s = 0; s < U.total; ++s) {
        const int g = gs0 + s, bb = g % C::NBUF, i = s / C::SPT, hh = s % C::SPT;
        const int gu = gq0 + C::unit_of(s), st = gu % C::NQS;
        // the step's U^T / dP^T, and the stage's per-query scalars (loaded long before)
        ok = __all_sync(0xffffffffu, mbar_wait_both(bar(B_S + bb), (g / C::NBUF) & 1,
                                                    bar(B_QF + st), (gu / C::NQS) & 1, ab));
        if (!ok) break;
        tc_fence_after();
        const float* sts = reinterpret_cast<const float*>(smem + C::OFF_STAT + st * C::STB);
        constexpr int CW = C::CW, H = CW / 16;
        const int cl = wg * CW;             // the warpgroup's columns within the step
        const int qt0 = hh * C::QW + cl;    // tile-local query index
        // Chunks of 16 queries (the next chunk's TMEM load in flight while one is
        // computed).  P (dS') of queries cl + 16 h .. go packed to columns cl + 8 h .. of
        // the U^T (dP^T) columns, which the first chunk has already read.
        uint32_t U0[16], G0[16], U1[16], G1[16];
        tmem_ld16(trow + C::col_u(bb) + cl, U0);
        tmem_ld16(trow + C::col_g(bb) + cl, G0);
        tmem_ld_wait();
        if (H > 1) {
          tmem_ld16(trow + C::col_u(bb) + cl + 16, U1);
          tmem_ld16(trow + C::col_g(bb) + cl + 16, G1);
        }
        uint32_t pk[CW / 2], dk[CW / 2];
        const float* stc = sts + (C::HALF ? cl : qt0);
        {
          uint32_t (&p0)[8] = *reinterpret_cast<uint32_t(*)[8]>(pk);
          uint32_t (&d0)[8] = *reinterpret_cast<uint32_t(*)[8]>(dk);
          if (i == 0)
            ew_chunk<true, C::SW, 16>(U0, G0, stc, qt0, t, kc, self2, p0, d0, dl2);
          else
            ew_chunk<false, C::SW, 16>(U0, G0, stc, qt0, t, kc, self2, p0, d0, dl2);
          tmem_st8(trow + C::col_u(bb) + cl, p0);  // P   (A operand of dV += P^T dO)
          tmem_st8(trow + C::col_g(bb) + cl, d0);  // dS' (A operand of dK += dS'^T Q)
        }
        if (H > 1) {
          tmem_ld_wait();
          uint32_t (&p1)[8] = *reinterpret_cast<uint32_t(*)[8]>(pk + 8 * (H - 1));
          uint32_t (&d1)[8] = *reinterpret_cast<uint32_t(*)[8]>(dk + 8 * (H - 1));
          if (i == 0)
            ew_chunk<true, C::SW, 16>(U1, G1, stc + 16, qt0 + 16, t, kc, self2, p1, d1, dl2);
          else
            ew_chunk<false, C::SW, 16>(U1, G1, stc + 16, qt0 + 16, t, kc, self2, p1, d1, dl2);
          tmem_st8(trow + C::col_u(bb) + cl + 8, p1);
          tmem_st8(trow + C::col_g(bb) + cl + 8, d1);
        }
        if (s == 0 && ul > 0) {
          // the previous unit's dK / dV staging, in the dS' buffer written next, has been
          // read by the stores of warpgroups 0 and 1 (every elementwise warp arrives)
          if (lane == 0) tma_store_wait_read_all();
          __syncwarp();
          mbar_arrive(bar(B_STG));
          ok = __all_sync(0xffffffffu, mbar_wait(bar(B_STG), (ul - 1) & 1, ab));
          if (!ok) break;
        }
        // dS' row t (key), the warpgroup's queries, into the 128-byte-swizzled query-major
        // layout the dQ product reads: 64-query blocks of 128 key rows
        uint8_t* ds_row = C::HALF ? smem + C::OFF_DS + (g & 1) * C::DSZ + t * 128
                                  : smem + C::OFF_DS + ((gt0 + i) & 1) * C::DSZ +
                                        (qt0 >> 6) * 16384 + t * 128;
        const int cb = (qt0 & 63) >> 3;
#pragma unroll
        for (int qd = 0; qd < CW / 8; ++qd)
          *reinterpret_cast<uint4*>(ds_row + (((cb + qd) ^ (t & 7)) << 4)) =
              make_uint4(dk[4 * qd], dk[4 * qd + 1], dk[4 * qd + 2], dk[4 * qd + 3]);
        tmem_st_wait();
        fence_async_smem();
        tc_fence_before();
        mbar_arrive(bar(B_P + bb));
      }
      if (!ok) break;
      // -------------------------------------------------- dK (warpgroup 0) / dV (1)
      // The sums over the unit's queries, Self entry included (diagonal of P and dS'):
      //   dK_j = (sum_i dS'_ij q_i) / (2 sqrt d),   dV_j = sum_i P_ij dO_i
      // (warpgroups 2 and 3 go on to the next unit)
      if (wg < 2) {
        if (!(ok = __all_sync(0xffffffffu, mbar_wait(bar(B_ACC), ul & 1, ab)))) break;
        tc_fence_after();
        const uint32_t col = wg == 0 ? C::COL_DK : C::COL_DV;
        const float sc = wg == 0 ? 0.5f * isd : 1.0f;
        // Staged as 32 rows x D per warp (128-byte swizzle) and written by TMA stores that
        // clip rows past T and padding columns.  d_h = 64: in the dS' buffer the next unit
        // writes first (its last reader, the dQ of the tile before last, precedes B_ACC);
        // d_h = 128 (one unit per CTA): in the Q (dK) and dO (dV) stages, which no MMA
        // reads any more.
        const uint32_t stg_off =
            (C::HALF ? (wg == 0 ? C::OFF_Q : C::OFF_DO)
                     : C::OFF_DS + ((gt0 + U.n_i) & 1) * C::DSZ + wg * (4 * 32 * D * 2)) +
            wq * (32 * D * 2);
        uint8_t* stg = smem + stg_off + lane * 128;
  #pragma unroll
        for (int c0 = 0; c0 < D; c0 += 32) {
          uint32_t a[32];
          tmem_ld32(trow + col + c0, a);
          tmem_ld_wait();
          const int kb = c0 >> 6;  // 64-column block
  #pragma unroll
          for (int c8 = 0; c8 < 32; c8 += 8) {
            uint32_t o4[4];
  #pragma unroll
            for (int e = 0; e < 4; ++e)
              o4[e] = pack_bf16x2(__uint_as_float(a[c8 + 2 * e]) * sc,
                                  __uint_as_float(a[c8 + 2 * e + 1]) * sc);
            const int chunk = ((c0 & 63) + c8) >> 3;  // 16-byte chunk within the 128-byte row
            *reinterpret_cast<uint4*>(stg + kb * (32 * 128) + ((chunk ^ (lane & 7)) << 4)) =
                make_uint4(o4[0], o4[1], o4[2], o4[3]);
          }
        }
        fence_async_smem();
        __syncwarp();
        if (lane == 0) {
          const CUtensorMap* tm = wg == 0 ? &tmDK : &tmDV;
  #pragma unroll
          for (int kb = 0; kb < C::KB; ++kb)
            tma_store_4d(tm, sb + stg_off + kb * (32 * 128), kb * 64, U.k0 + wq * 32, U.h, U.b);
          tma_store_commit();  // its reads are awaited before the staging is written again
        }
        __syncwarp();
      }
      gs0 += U.total;
      gq0 += U.n_units;
      gt0 += U.n_i;
    }
    if (lane == 0) tma_store_wait_read_all();  // the staging must outlive the store's reads
    float dlam = dl2.x + dl2.y;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dlam += __shfl_xor_sync(0xffffffffu, dlam, o);
    if (lane == 0) red[warp] = dlam;
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < C::EW_THREADS / 32; ++w) s += red[w];
    ws.dlam_part[ws.n_pre_blocks + blockIdx.x] = s;
  }
  if (warp == C::W_MMA) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Row pass over the padded rows r < t_pad of every head, 8 threads per row:
//   D_i = dO_i . Y_i,  g_ii = dO_i . v_i,  S_i = sigmoid(u_ii / tau_S),
//   F_ii = exp(S_i - logZ_i) (the Self flow),
//   Self entry: dR_ii = F_ii (g_ii - D_i),  dS_ii = dR_ii S_i (1 - S_i) / tau_S
//   (F_self, dS_self for the tile kernel's diagonal) and its dlambda term log i (1 - F_ii) dR_ii
//   (one partial per block);
// the per-query scalars of the tile kernel (three arrays per 128-row tile:
// c2 = (-lambda log i - logZ_i) log2 e, -D_i, -log i F_ii) and a zeroed row of the fp32 dQ
// accumulator.  Padding rows get neutral scalars (P = 0).
template <int D>
__global__ void __launch_bounds__(256) pre_kernel(Problem p, BwdWorkspace ws, int n_t) {
  __shared__ float part[8];
  constexpr int PER = D / 8;  // elements per thread
  const long long gr = ((long long)blockIdx.x * 256 + threadIdx.x) >> 3;
  const int sub = threadIdx.x & 7;
  const long long nrows = (long long)p.B * p.H * ws.t_pad;
  const bool live = gr < nrows;
  const long long grc = live ? gr : 0;
  const int bh = (int)(grc / ws.t_pad), r = (int)(grc % ws.t_pad);
  const bool real = live && r < p.T;
  const int b = bh / p.H, h = bh % p.H;
  const long long off = (long long)b * p.sB + (long long)h * p.sH + (long long)r * p.sT + sub * PER;
  float gy = 0.f, gv = 0.f, qk = 0.f;
  if (real) {
    auto bf = [](const void* base, long long o) {
      return *reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(base) + o);
    };
#pragma unroll
    for (int c = 0; c < PER; c += 8) {
      if (sub * PER + c >= p.d) break;  // padding columns (d_h < D)
      const uint4 gv4 = bf(p.dout, off + c), ov = bf(p.o, off + c), vv = bf(p.v, off + c);
      const uint4 qv = bf(p.q, off + c), kv = bf(p.k, off + c);
      const uint32_t g4[4] = {gv4.x, gv4.y, gv4.z, gv4.w}, o4[4] = {ov.x, ov.y, ov.z, ov.w};
      const uint32_t v4[4] = {vv.x, vv.y, vv.z, vv.w};
      const uint32_t q4[4] = {qv.x, qv.y, qv.z, qv.w}, k4[4] = {kv.x, kv.y, kv.z, kv.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 gf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&g4[e]));
        const float2 of = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&o4[e]));
        const float2 vf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&v4[e]));
        const float2 qf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&q4[e]));
        const float2 kf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&k4[e]));
        gy = fmaf(gf.x, of.x, fmaf(gf.y, of.y, gy));
        gv = fmaf(gf.x, vf.x, fmaf(gf.y, vf.y, gv));
        qk = fmaf(qf.x, kf.x, fmaf(qf.y, kf.y, qk));
      }
    }
  }
#pragma unroll
  for (int o = 4; o > 0; o >>= 1) {
    gy += __shfl_xor_sync(0xffffffffu, gy, o);
    gv += __shfl_xor_sync(0xffffffffu, gv, o);
    qk += __shfl_xor_sync(0xffffffffu, qk, o);
  }
  float contrib = 0.f;
  if (live && sub == 0) {
    float c2 = -INFINITY, nd = 0.f, nw = 0.f;
    if (real) {
      const long long srow = (long long)bh * p.T + r;
      const float lz = p.logz_in[srow];
      const float li = logf((float)(r + 1));
      const float S = 1.0f / (1.0f + expf(-(qk * p.inv_sqrt_d) / p.tau_s));
      const float F = expf(S - lz);
      const float dR = F * (gv - gy);
      ws.F_self[srow] = F;
      ws.dS_self[srow] = dR * S * (1.0f - S) / p.tau_s;
      contrib = li * (1.0f - F) * dR;
      c2 = (-p.lambda * li - lz) * kLog2e;
      nd = -gy;
      nw = -li * F;
    }
    float* st = ws.stats + ((long long)bh * n_t + (r >> 7)) * 3 * BT + (r & 127);
    st[0] = c2;
    st[BT] = nd;
    st[2 * BT] = nw;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) contrib += __shfl_xor_sync(0xffffffffu, contrib, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = contrib;
  if (live) {
    float* acc = ws.dq_acc + ((long long)bh * ws.t_pad + r) * D + sub * PER;
#pragma unroll
    for (int c = 0; c < PER; c += 4)
      *reinterpret_cast<float4*>(acc + c) = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) t += part[w];
    ws.dlam_part[blockIdx.x] = t;
  }
}

// dq = bf16(dq_acc / (2 sqrt(d))) for rows < T (the accumulator holds the Exchange sums
// and the Self entry, which the diagonal tile carries); block 0 also reduces the dlambda
// partials of the row pass (n_pre) and of the tile kernel (n_cta) in a fixed order
// (deterministic).
template <int D>
__global__ void __launch_bounds__(256) finalize_kernel(Problem p, BwdWorkspace ws, int n_pre,
                                                       int n_cta) {
  if (blockIdx.x == 0) {
    __shared__ double part[256];
    double s = 0.0;
    for (int i = threadIdx.x; i < n_pre; i += 256) s += (double)ws.dlam_part[i];
    for (int i = threadIdx.x; i < n_cta; i += 256) s += (double)ws.dlam_part[ws.n_pre_blocks + i];
    part[threadIdx.x] = s;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
      if (threadIdx.x < w) part[threadIdx.x] += part[threadIdx.x + w];
      __syncthreads();
    }
    if (threadIdx.x == 0) *p.dlambda = (float)part[0];
  }
  const long long idx = ((long long)blockIdx.x * 256 + threadIdx.x);  // 8-wide chunk
  const long long per_row = p.d / 8;  // 8-column chunks of the real columns
  const long long n = (long long)p.B * p.H * p.T * per_row;
  if (idx >= n) return;
  const int c8 = (int)(idx % per_row) * 8;
  const long long row = idx / per_row;
  const int bh = (int)(row / p.T), r = (int)(row % p.T);
  const int b = bh / p.H, h = bh % p.H;
  const float* src = ws.dq_acc + ((long long)bh * ws.t_pad + r) * D + c8;
  const float4 a = *reinterpret_cast<const float4*>(src);
  const float4 c = *reinterpret_cast<const float4*>(src + 4);
  const long long off = (long long)b * p.sB + (long long)h * p.sH + (long long)r * p.sT + c8;
  const float sc = 0.5f * p.inv_sqrt_d;
  uint4 o;
  o.x = pack_bf16x2(a.x * sc, a.y * sc);
  o.y = pack_bf16x2(a.z * sc, a.w * sc);
  o.z = pack_bf16x2(c.x * sc, c.y * sc);
  o.w = pack_bf16x2(c.z * sc, c.w * sc);
  *reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(p.dq) + off) = o;
}

}  // namespace bwd

// 2-D map over the fp32 dQ accumulator [B*H*t_pad][D]: box 32 x 32, 128-byte swizzle.
static bool make_tmap_dq(CUtensorMap* m, float* base, int rows, int d) {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return false;
    fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)d * 4};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tile-kernel CTAs.  d_h <= 64: persistent, one CTA per SM over the (key tile, head)
// units; d_h = 128 stages dK / dV in its Q / dO stages and takes one unit per CTA.
static long long tile_grid(const Problem& p) {
  const long long units = (long long)((p.T + 127) / 128) * p.B * p.H;
  if (p.d > 64) return units;
  int dev = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || nsm < 1)
    return units;
  return units < nsm ? units : nsm;
}

template <int D>
static cudaError_t bwd_t(const Problem& p, const BwdWorkspace& ws, unsigned stages,
                         cudaStream_t s) {
  const int n_t = (p.T + 127) / 128;
  const int t_pad = ws.t_pad;
  const long long rows = (long long)p.B * p.H * p.T;
  if ((long long)n_t * p.B * p.H > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  const long long grid = tile_grid(p);
  cudaError_t e = cudaSuccess;
  if (stages & 1) {
    const long long rows_pad = (long long)p.B * p.H * t_pad;
    bwd::pre_kernel<D><<<(unsigned)((rows_pad * 8 + 255) / 256), 256, 0, s>>>(p, ws, n_t);
    if ((e = cudaGetLastError()) != cudaSuccess) { note_failure("backward: row pass launch"); return e; }
  }
  if (stages & 2) {
    // A runtime call first: it makes the device's primary context current on this thread,
    // which the driver's tensor-map encoder needs (e.g. on a fresh autograd worker thread).
    const int smem = bwd::Cfg<D>::SMEM;
    e = cudaFuncSetAttribute(bwd::bwd_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem);
    if (e != cudaSuccess) { note_failure("backward: shared memory attribute"); return e; }
    CUtensorMap mq, mk, mv, mg, mdq, mdk, mdv;
    constexpr int qrows = bwd::Cfg<D>::QROWS;
    if (!make_tmap_bf16(&mq, p.q, p, qrows) || !make_tmap_bf16(&mk, p.k, p, 128) ||
        !make_tmap_bf16(&mv, p.v, p, 128) || !make_tmap_bf16(&mg, p.dout, p, qrows) ||
        !make_tmap_bf16(&mdk, p.dk, p, 32) || !make_tmap_bf16(&mdv, p.dv, p, 32)) {
      note_failure("backward: TMA descriptor of Q/K/V/dO/dK/dV");
      return cudaErrorInvalidValue;
    }
    if (!make_tmap_dq(&mdq, ws.dq_acc, p.B * p.H * t_pad, D)) {
      note_failure("backward: TMA descriptor of the dQ accumulator");
      return cudaErrorInvalidValue;
    }
    int dev = 0, nsm = 148;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      nsm = 148;
    // d_h = 128 (one CTA per unit, dynamic scheduling): heads in groups, one CTA per SM;
    // d_h = 64 (persistent, zigzag over a heaviest-first sequence): one group.
    const int groups = D == 64 ? 1 : head_groups(n_t, p.B * p.H, nsm);
    bwd::bwd_tc_kernel<D><<<(unsigned)grid, bwd::Cfg<D>::THREADS, smem, s>>>(mq, mk, mv, mg, mdq, mdk,
                                                                     mdv, p, ws, n_t, t_pad, groups);
    if ((e = cudaGetLastError()) != cudaSuccess) { note_failure("backward: tile kernel launch"); return e; }
  }
  if (stages & 4) {
    const long long chunks = rows * (p.d / 8);
    const long long fblocks = (chunks + 255) / 256;
    const int n_pre = (int)((long long)p.B * p.H * t_pad / 32);  // row-pass blocks
    bwd::finalize_kernel<D><<<(unsigned)(fblocks > 0 ? fblocks : 1), 256, 0, s>>>(p, ws, n_pre,
                                                                                (int)grid);
    if ((e = cudaGetLastError()) != cudaSuccess) note_failure("backward: finalisation launch");
  }
  return e;
}

bool supports_bwd(relation_dtype dt, int d) { return supports(dt, d); }

cudaError_t launch_bwd(const Problem& p, const BwdWorkspace& ws, unsigned stages,
                       cudaStream_t s) {
  if (!supports_bwd(p.dtype, p.d)) return cudaErrorInvalidValue;
  return p.d <= 64 ? bwd_t<64>(p, ws, stages, s) : bwd_t<128>(p, ws, stages, s);
}
int bwd_launches() { return 3; }
int main_ctas(const Problem& p) { return ((p.T + 127) / 128) * p.B * p.H; }

}  // namespace tc
}  // namespace rel
