// relation_tc_bwd.cu -- tcgen05 / TMA / TMEM backward of FlashRelation (bf16, d_h 64/128).
//
// Gradient (App. A.1.7, generic softmax form) for the Exchange pairs j < i:
//   P_ij  = exp(E_ij - lambda log i - logZ_i)        (recomputed; F_ij of the flow)
//   dP_ij = dO_i . v_j,   dR_ij = P_ij (dP_ij - D_i)
//   dS_ij = dR_ij SiLU'(u_ij),  SiLU'(u) = sigma(u) + u sigma(u) (1 - sigma(u))
//   dV_j += P_ij dO_i,  dK_j += dS_ij q_i / sqrt(d),  dQ_i += dS_ij k_j / sqrt(d)
// The Self pairs (j = i), D_i and the initial value of the fp32 dQ accumulator come from
// the row pre-pass (aux_kernels.cu); a finalisation kernel converts dQ to bf16.
//
// One CTA owns a tile of 128 keys of one head and visits the query tiles from its
// diagonal tile to the end of the sequence.  Per query tile, with keys on TMEM lanes:
//   MMA  U^T  = K Q^T,  dP^T = V dO^T                  (TMEM, fp32)
//   elementwise (warps 0-3, thread = key): P and dS' = 2 dS in bf16; P into TMEM,
//        dS' into shared memory (128-byte swizzled rows of 128 queries)
//   MMA  dV += P^T dO (P from TMEM),  dK += dS'^T Q,  dQ_i = dS' K
//   warps 4-7 read dQ_i (queries on lanes) and add it to the fp32 accumulator.
// Warp 8 loads tiles with TMA and stages the per-query scalars; warp 9 issues MMAs.
// The factor 1/2 of dS' and 1/sqrt(d) are applied in the fp32 epilogues.  dL/dlambda's
// Exchange part  -sum log i F_ii dR_ij  is accumulated per key and reduced per CTA.
#include <cudaTypedefs.h>
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rel {
namespace tc {

namespace bwd {

constexpr int BK = 128;         // keys per CTA
constexpr int BQ = 128;         // queries per step
constexpr int kThreads = 320;   // 4 elementwise + 4 dQ + TMA + MMA warps
constexpr int kTmemCols = 512;

template <int D>
struct Cfg {
  static constexpr int KB = D / 64;
  static constexpr int TILE = 128 * D * 2;           // bytes of a K, V, Q or dO tile
  static constexpr int QS = D == 64 ? 2 : 1;         // Q / dO stages
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = OFF_K + TILE;
  static constexpr int OFF_Q = OFF_V + TILE;
  static constexpr int OFF_DO = OFF_Q + QS * TILE;
  static constexpr int OFF_DS = OFF_DO + QS * TILE;  // 128 keys x 128 queries bf16
  static constexpr int OFF_STAT = OFF_DS + BK * BQ * 2;
  static constexpr int STAT_STAGE = 3 * BQ * 4;      // c2, D, w per query
  static constexpr int OFF_RED = OFF_STAT + QS * STAT_STAGE;
  static constexpr int OFF_BAR = OFF_RED + 64;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static constexpr int COL_ST = 0, COL_DPT = 128, COL_DK = 256, COL_DV = 256 + D;
  static constexpr int COL_DQ = D == 64 ? 384 : 128;  // d=128: reuses the dP^T columns
};

enum : int {
  B_KV = 0, B_QF = 1, B_QE = 3, B_S = 5, B_P = 6, B_DQF = 7, B_DQE = 8, B_ACC = 9
};

__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > 20ull * 1000ull * 1000ull) return;
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    bwd_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmG,
                  Problem p, BwdWorkspace ws, int n_t, int t_pad) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sb = smem_u32(smem);
  auto bar = [&](int i) -> uint32_t { return sb + C::OFF_BAR + 8u * (uint32_t)i; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_BAR + 128);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_BAR + 136);
  float* red = reinterpret_cast<float*>(smem + C::OFF_RED);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int BH = p.B * p.H;
  const int kt = (int)(blockIdx.x / BH);  // heaviest key tiles (most query tiles) first
  const int bh = (int)(blockIdx.x % BH);
  const int b = bh / p.H, h = bh % p.H;
  const int k0 = kt * BK;
  const int n_i = n_t - kt;  // query tiles kt .. n_t - 1

  if (threadIdx.x == 0) {
    mbar_init(bar(B_KV), 1);
    for (int s = 0; s < C::QS; ++s) {
      mbar_init(bar(B_QF + s), 1);
      mbar_init(bar(B_QE + s), 1);
    }
    mbar_init(bar(B_S), 1);
    mbar_init(bar(B_P), 128);
    mbar_init(bar(B_DQF), 1);
    mbar_init(bar(B_DQE), 128);
    mbar_init(bar(B_ACC), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 9) tmem_alloc(smem_u32(tmem_slot), kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const Abort ab{abort_flag, p.dev_status};
  const long long rows_bh = (long long)bh * p.T;

  if (warp == 8) {
    // ---------------------------------------------------------- TMA + per-query scalars
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmG);
      mbar_arrive_expect_tx(bar(B_KV), 2 * C::TILE);
      for (int kb = 0; kb < C::KB; ++kb) {
        tma_load_4d(sb + C::OFF_K + kb * 128 * 128, &tmK, bar(B_KV), kb * 64, k0, h, b);
        tma_load_4d(sb + C::OFF_V + kb * 128 * 128, &tmV, bar(B_KV), kb * 64, k0, h, b);
      }
    }
    int issued = 0;
    for (int i = 0; i < n_i; ++i) {
      const int s = i % C::QS, u = i / C::QS;
      bool ok = true;
      if (u > 0) ok = mbar_wait(bar(B_QE + s), (u - 1) & 1, ab);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      const int qi0 = (kt + i) * BQ;
      float* st = reinterpret_cast<float*>(smem + C::OFF_STAT + s * C::STAT_STAGE);
      for (int q = lane; q < BQ; q += 32) {
        const int row = qi0 + q;
        float c2 = -INFINITY, dd = 0.f, wl = 0.f;
        if (row < p.T) {
          const float li = __logf((float)(row + 1));
          c2 = (-p.lambda * li - p.logz_in[rows_bh + row]) * kLog2e;
          dd = ws.D[rows_bh + row];
          wl = li * ws.F_self[rows_bh + row];
        }
        st[q] = c2;
        st[BQ + q] = dd;
        st[2 * BQ + q] = wl;
      }
      __threadfence_block();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive_expect_tx(bar(B_QF + s), 2 * C::TILE);
        for (int kb = 0; kb < C::KB; ++kb) {
          tma_load_4d(sb + C::OFF_Q + s * C::TILE + kb * 128 * 128, &tmQ, bar(B_QF + s),
                      kb * 64, qi0, h, b);
          tma_load_4d(sb + C::OFF_DO + s * C::TILE + kb * 128 * 128, &tmG, bar(B_QF + s),
                      kb * 64, qi0, h, b);
        }
      }
      issued = i + 1;
    }
    if (lane == 0 && ab.raised()) {
      drain_wait(bar(B_KV), 0);
      for (int i = issued - C::QS > 0 ? issued - C::QS : 0; i < issued; ++i)
        drain_wait(bar(B_QF + i % C::QS), (i / C::QS) & 1);
    }
  } else if (warp == 9) {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t id_qk = idesc_bf16_f32(128, 128, false, false);  // U^T, dP^T
      constexpr uint32_t id_acc = idesc_bf16_f32(128, D, false, true);    // dV, dK
      constexpr uint32_t id_dq = idesc_bf16_f32(128, D, true, true);      // dQ
      auto issue_scores = [&](int s) {
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t koff = (kk >> 2) * (128 * 128) + (kk & 3) * 32;
          mma_ss(tmem + C::COL_ST, smem_desc_sw128(sb + C::OFF_K + koff, 16, 1024),
                 smem_desc_sw128(sb + C::OFF_Q + s * C::TILE + koff, 16, 1024), id_qk,
                 kk > 0 ? 1u : 0u);
        }
      };
      auto issue_dp = [&](int s) {
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t koff = (kk >> 2) * (128 * 128) + (kk & 3) * 32;
          mma_ss(tmem + C::COL_DPT, smem_desc_sw128(sb + C::OFF_V + koff, 16, 1024),
                 smem_desc_sw128(sb + C::OFF_DO + s * C::TILE + koff, 16, 1024), id_qk,
                 kk > 0 ? 1u : 0u);
        }
      };
      bool ok = mbar_wait(bar(B_KV), 0, ab) && mbar_wait(bar(B_QF), 0, ab);
      tc_fence_after();
      if (ok) {
        issue_scores(0);
        issue_dp(0);
        mma_commit(bar(B_S));
      }
      for (int i = 0; ok && i < n_i; ++i) {
        const int s = i % C::QS;
        if (!(ok = mbar_wait(bar(B_P), i & 1, ab))) break;
        tc_fence_after();
        const uint32_t acc0 = i > 0 ? 1u : 0u;
        // dV += P^T dO_i   (A = P^T from TMEM; B = dO tile, N = d contiguous)
#pragma unroll
        for (int kk = 0; kk < BQ / 16; ++kk)
          mma_ts(tmem + C::COL_DV, tmem + C::COL_ST + kk * 8,
                 smem_desc_sw128(sb + C::OFF_DO + s * C::TILE + kk * 2048, 128 * 128, 1024),
                 id_acc, (acc0 | (kk > 0)) ? 1u : 0u);
        // dK += dS'^T Q_i   (A = dS'^T: keys x queries, queries contiguous)
#pragma unroll
        for (int kk = 0; kk < BQ / 16; ++kk)
          mma_ss(tmem + C::COL_DK,
                 smem_desc_sw128(sb + C::OFF_DS + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                 smem_desc_sw128(sb + C::OFF_Q + s * C::TILE + kk * 2048, 128 * 128, 1024),
                 id_acc, (acc0 | (kk > 0)) ? 1u : 0u);
        if (D == 64 && i > 0) {
          if (!(ok = mbar_wait(bar(B_DQE), (i - 1) & 1, ab))) break;
          tc_fence_after();
        }
        // dQ_i = dS' K   (A = dS': queries x keys, queries contiguous; B = K tile)
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk)
          mma_ss(tmem + C::COL_DQ, smem_desc_sw128(sb + C::OFF_DS + kk * 2048, 16384, 1024),
                 smem_desc_sw128(sb + C::OFF_K + kk * 2048, 128 * 128, 1024), id_dq,
                 kk > 0 ? 1u : 0u);
        mma_commit(bar(B_DQF));
        mma_commit(bar(B_QE + s));
        if (i + 1 < n_i) {
          const int s1 = (i + 1) % C::QS, u1 = (i + 1) / C::QS;
          if (!(ok = mbar_wait(bar(B_QF + s1), u1 & 1, ab))) break;
          tc_fence_after();
          issue_scores(s1);
          if (D == 128) {
            if (!(ok = mbar_wait(bar(B_DQE), i & 1, ab))) break;
            tc_fence_after();
          }
          issue_dp(s1);
          mma_commit(bar(B_S));
        }
      }
      mma_commit(bar(B_ACC));
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ---------------------------------------------------------- dQ_i -> fp32 accumulator
    const int q = (warp - 4) * 32 + lane;
    const uint32_t trow = tmem + ((uint32_t)((warp - 4) * 32) << 16);
    for (int i = 0; i < n_i; ++i) {
      const bool ok = __all_sync(0xffffffffu, mbar_wait(bar(B_DQF), i & 1, ab));
      if (!ok) break;
      tc_fence_after();
      const int row = (kt + i) * BQ + q;
      float* dst = ws.dq_acc + ((long long)bh * t_pad + row) * D;
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32) {
        uint32_t z[32];
        tmem_ld32(trow + C::COL_DQ + c0, z);
        tmem_ld_wait();
        if (row < p.T) {
#pragma unroll
          for (int c = 0; c < 32; c += 4)
            atomicAdd(reinterpret_cast<float4*>(dst + c0 + c),
                      make_float4(__uint_as_float(z[c]), __uint_as_float(z[c + 1]),
                                  __uint_as_float(z[c + 2]), __uint_as_float(z[c + 3])));
        }
      }
      tc_fence_before();
      mbar_arrive(bar(B_DQE));
    }
  } else {
    // ---------------------------------------------------------- elementwise + epilogue
    const int t = threadIdx.x;  // key k0 + t, TMEM lane t
    const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
    const float isd = p.inv_sqrt_d;
    const float ch = 0.5f * isd;   // h = U ch = u / 2
    const float c2k = ch * kLog2e; // E log2 e = U c2k (1 + tanh h)
    uint8_t* ds_row = smem + C::OFF_DS + t * 128;
    const int sw = t & 7;
    float dlam = 0.f;
    bool ok = true;
    for (int i = 0; i < n_i; ++i) {
      const int s = i % C::QS;
      ok = __all_sync(0xffffffffu, mbar_wait(bar(B_S), i & 1, ab));
      if (!ok) break;
      tc_fence_after();
      const float* st = reinterpret_cast<const float*>(smem + C::OFF_STAT + s * C::STAT_STAGE);
      const bool diag = (i == 0);
#pragma unroll 1
      for (int c0 = 0; c0 < BQ; c0 += 32) {
        uint32_t U[32], G[32];
        tmem_ld32(trow + C::COL_ST + c0, U);
        tmem_ld32(trow + C::COL_DPT + c0, G);
        tmem_ld_wait();
        uint32_t pk[16], dk[16];
#pragma unroll
        for (int c = 0; c < 32; c += 4) {
          const float4 c2v = *reinterpret_cast<const float4*>(st + c0 + c);
          const float4 ddv = *reinterpret_cast<const float4*>(st + BQ + c0 + c);
          const float4 wlv = *reinterpret_cast<const float4*>(st + 2 * BQ + c0 + c);
          const float c2a[4] = {c2v.x, c2v.y, c2v.z, c2v.w};
          const float dda[4] = {ddv.x, ddv.y, ddv.z, ddv.w};
          const float wla[4] = {wlv.x, wlv.y, wlv.z, wlv.w};
          float pv[4], dv[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int col = c0 + c + e;
            const float x = __uint_as_float(U[c + e]);
            const float hh = x * ch;
            const float th = tanh_approx(hh);
            const float w = fmaf(th, c2k, c2k);
            float P = ex2_approx(fmaf(x, w, c2a[e]));
            if (diag && col <= t) P = 0.f;  // history only: query > key
            const float dR = P * (__uint_as_float(G[c + e]) - dda[e]);
            // 2 SiLU'(u) = 1 + t + h (1 - t^2) with t = tanh(u/2), h = u/2
            const float sp = 1.0f + th + fmaf(-hh * th, th, hh);
            dlam = fmaf(-wla[e], dR, dlam);
            pv[e] = P;
            dv[e] = dR * sp;
          }
          pk[c >> 1] = pack_bf16x2(pv[0], pv[1]);
          pk[(c >> 1) + 1] = pack_bf16x2(pv[2], pv[3]);
          dk[c >> 1] = pack_bf16x2(dv[0], dv[1]);
          dk[(c >> 1) + 1] = pack_bf16x2(dv[2], dv[3]);
        }
        tmem_st16(trow + C::COL_ST + (c0 >> 1), pk);
        // dS' row t, queries c0..c0+31: 4 chunks of 16 bytes in the 128-byte swizzle
        const int atom = c0 >> 6, cb = (c0 & 63) >> 3;
#pragma unroll
        for (int qd = 0; qd < 4; ++qd) {
          const int phys = (cb + qd) ^ sw;
          *reinterpret_cast<uint4*>(ds_row + atom * 16384 + phys * 16) =
              make_uint4(dk[4 * qd], dk[4 * qd + 1], dk[4 * qd + 2], dk[4 * qd + 3]);
        }
      }
      tmem_st_wait();
      fence_async_smem();
      tc_fence_before();
      mbar_arrive(bar(B_P));
    }
    // ------------------------------------------------------------ dK, dV epilogue
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar(B_ACC), 0, ab));
    tc_fence_after();
    if (ok) {
      const int j = k0 + t;
      const long long off = (long long)b * p.sB + (long long)h * p.sH + (long long)j * p.sT;
      const __nv_bfloat16* qrow = reinterpret_cast<const __nv_bfloat16*>(p.q) + off;
      const __nv_bfloat16* grow = reinterpret_cast<const __nv_bfloat16*>(p.dout) + off;
      __nv_bfloat16* dkrow = reinterpret_cast<__nv_bfloat16*>(p.dk) + off;
      __nv_bfloat16* dvrow = reinterpret_cast<__nv_bfloat16*>(p.dv) + off;
      const bool valid = j < p.T;
      const float fs = valid ? ws.F_self[rows_bh + j] : 0.f;
      const float dss = valid ? ws.dS_self[rows_bh + j] : 0.f;
#pragma unroll 1
      for (int c0 = 0; c0 < D; c0 += 32) {
        uint32_t ak[32], av[32];
        tmem_ld32(trow + C::COL_DK + c0, ak);
        tmem_ld32(trow + C::COL_DV + c0, av);
        tmem_ld_wait();
        if (valid) {
#pragma unroll
          for (int c8 = 0; c8 < 32; c8 += 8) {
            const uint4 qv = *reinterpret_cast<const uint4*>(qrow + c0 + c8);
            const uint4 gv = *reinterpret_cast<const uint4*>(grow + c0 + c8);
            const uint32_t qw[4] = {qv.x, qv.y, qv.z, qv.w};
            const uint32_t gw[4] = {gv.x, gv.y, gv.z, gv.w};
            uint32_t ok4[4], ov4[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 qf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qw[e]));
              const float2 gf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&gw[e]));
              const int c = c8 + 2 * e;
              const float k0f = fmaf(0.5f, __uint_as_float(ak[c]), dss * qf.x) * isd;
              const float k1f = fmaf(0.5f, __uint_as_float(ak[c + 1]), dss * qf.y) * isd;
              const float v0f = fmaf(fs, gf.x, __uint_as_float(av[c]));
              const float v1f = fmaf(fs, gf.y, __uint_as_float(av[c + 1]));
              ok4[e] = pack_bf16x2(k0f, k1f);
              ov4[e] = pack_bf16x2(v0f, v1f);
            }
            *reinterpret_cast<uint4*>(dkrow + c0 + c8) = make_uint4(ok4[0], ok4[1], ok4[2], ok4[3]);
            *reinterpret_cast<uint4*>(dvrow + c0 + c8) = make_uint4(ov4[0], ov4[1], ov4[2], ov4[3]);
          }
        }
      }
    }
    // per-warp dlambda partial
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dlam += __shfl_xor_sync(0xffffffffu, dlam, o);
    if (lane == 0) red[warp] = dlam;
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0)
    ws.dlam_part[ws.n_pre_blocks + blockIdx.x] = (red[0] + red[1]) + (red[2] + red[3]);
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// dq = bf16(dq_acc / (2 sqrt(d))) for rows < T  (dq_acc holds 2 x the unscaled sum)
template <int D>
__global__ void __launch_bounds__(256) dq_finalize_kernel(Problem p, const float* dq_acc,
                                                          int t_pad) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;  // 8-wide chunk
  const long long per_row = D / 8;
  const long long n = (long long)p.B * p.H * p.T * per_row;
  if (idx >= n) return;
  const int c8 = (int)(idx % per_row) * 8;
  const long long row = idx / per_row;  // over B*H*T
  const int bh = (int)(row / p.T), r = (int)(row % p.T);
  const int b = bh / p.H, h = bh % p.H;
  const float* src = dq_acc + ((long long)bh * t_pad + r) * D + c8;
  const float4 a = *reinterpret_cast<const float4*>(src);
  const float4 c = *reinterpret_cast<const float4*>(src + 4);
  const float sc = 0.5f * p.inv_sqrt_d;
  uint4 o;
  o.x = pack_bf16x2(a.x * sc, a.y * sc);
  o.y = pack_bf16x2(a.z * sc, a.w * sc);
  o.z = pack_bf16x2(c.x * sc, c.y * sc);
  o.w = pack_bf16x2(c.z * sc, c.w * sc);
  __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(p.dq) + (long long)b * p.sB +
                       (long long)h * p.sH + (long long)r * p.sT + c8;
  *reinterpret_cast<uint4*>(dst) = o;
}

}  // namespace bwd

bool make_tmap_bf16(CUtensorMap* m, const void* base, const Problem& p, int rows);

template <int D>
static cudaError_t bwd_t(const Problem& p, const BwdWorkspace& ws, cudaStream_t s) {
  CUtensorMap mq, mk, mv, mg;
  if (!make_tmap_bf16(&mq, p.q, p, 128) || !make_tmap_bf16(&mk, p.k, p, 128) ||
      !make_tmap_bf16(&mv, p.v, p, 128) || !make_tmap_bf16(&mg, p.dout, p, 128))
    return cudaErrorInvalidValue;
  const int smem = bwd::Cfg<D>::SMEM;
  cudaError_t e = cudaFuncSetAttribute(bwd::bwd_tc_kernel<D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int n_t = (p.T + 127) / 128;
  const int t_pad = n_t * 128;
  const long long grid = (long long)n_t * p.B * p.H;
  if (grid > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  bwd::bwd_tc_kernel<D><<<(unsigned)grid, bwd::kThreads, smem, s>>>(mq, mk, mv, mg, p, ws, n_t,
                                                                   t_pad);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const long long chunks = (long long)p.B * p.H * p.T * (D / 8);
  bwd::dq_finalize_kernel<D><<<(unsigned)((chunks + 255) / 256), 256, 0, s>>>(p, ws.dq_acc, t_pad);
  return cudaGetLastError();
}

bool supports_bwd(relation_dtype dt, int d) { return dt == RELATION_BF16 && (d == 64 || d == 128); }

cudaError_t launch_bwd(const Problem& p, const BwdWorkspace& ws, cudaStream_t s) {
  if (p.d == 64) return bwd_t<64>(p, ws, s);
  if (p.d == 128) return bwd_t<128>(p, ws, s);
  return cudaErrorInvalidValue;
}
int bwd_launches() { return 2; }
int main_ctas(const Problem& p) { return ((p.T + 127) / 128) * p.B * p.H; }

}  // namespace tc
}  // namespace rel
