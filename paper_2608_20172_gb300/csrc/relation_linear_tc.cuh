// relation_linear_tc.cuh -- shared pieces of the chunked tensor-core Linear Relation
// kernels (relation_linear_tc.cu: forward, state scans; relation_linear_tc_bwd.cu:
// backward): block size, the workspace view, shared-memory layout helpers, tensor maps.
#pragma once

#include <cudaTypedefs.h>
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rel {
namespace tc {
bool make_tmap_bf16(CUtensorMap* m, const void* base, const Problem& p, int rows);
}
namespace lintc {


constexpr int LT = 128;          // tokens per block
constexpr int NC = 64;           // information columns per CTA
constexpr int kThreads = 192;    // warps 0-3 elementwise, 4 TMA, 5 MMA
constexpr int kTmemCols = 256;   // S 128 | E 64 | C 64
constexpr int COL_S = 0, COL_E = 128, COL_C = 192;
constexpr float kClampLog2 = 120.0f;

// Modes of the kernel: SEQ walks all blocks of a (head, split) in order with the state in
// TMEM; the chunk-parallel pair takes one block per CTA: DELTA writes the block's state
// contribution sum_j KL_j I~_j^T and decay a_L (fp32) to the workspace, OUT reads the
// state the block starts from (bf16, produced by scan_kernel) and writes the block's Y.
// BDELTA is DELTA for the backward: the block's contribution to the state's adjoint,
// Qs^T dY (Qs in KL's place, dY in I~'s).
enum : int { MODE_SEQ = 0, MODE_DELTA = 1, MODE_OUT = 2, MODE_BDELTA = 3 };

// Workspace of the chunk-parallel forward, per (head, split, block): dC [D][64] fp32, the
// decay g [D] fp32, and per (head, split) nb + 1 states C0 [D][64] bf16 (the state entering
// every block, then the final one).
struct LinCp {
  float* dC;
  float* g;
  __nv_bfloat16* c0;
  int nb;
};

// B_LOAD, B_FREE, B_EPI: one per input stage (stage s at + s)
enum : int { B_LOAD = 0, B_FREE = 2, B_EPI = 4, B_OPS = 6, B_C0, B_S, B_A, B_E, B_STATE, NBAR };

__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > 20ull * 1000ull * 1000ull) return;
  }
}
// 2-D tiled load into shared memory, completing on `bar` (transaction bytes).
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* m, uint32_t bar,
                                            int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), "r"(c0), "r"(c1)
      : "memory");
}
__device__ __forceinline__ void ew_sync() {  // the 128 elementwise threads
  asm volatile("bar.sync 1, 128;" ::: "memory");
}
// byte offset of element (row r, column c) in a tile of 128-byte-swizzled rows of 64
// bf16 columns, blocks of `rows` rows per 64 columns
__device__ __forceinline__ uint32_t swz(int r, int c, int rows) {
  return (uint32_t)((c >> 6) * rows * 128 + r * 128 + ((((c & 63) >> 3) ^ (r & 7)) << 4) +
                    (c & 7) * 2);
}
// element (token, channel) of [d / 32][128][32] fp32 tiles written by the swizzled
// retention map: the 16-byte groups of a token's 128-byte row permuted by (token & 7)
__device__ __forceinline__ int al_swz(int tok, int ch) {
  return (ch >> 5) * (LT * 32) + tok * 32 + ((((ch & 31) >> 2) ^ (tok & 7)) << 2) + (ch & 3);
}
__device__ __forceinline__ float ld_bf(const uint8_t* base, uint32_t off) {
  return __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(base + off));
}
__device__ __forceinline__ void st_bf(uint8_t* base, uint32_t off, float x) {
  *reinterpret_cast<__nv_bfloat16*>(base + off) = __float2bfloat16_rn(x);
}


// 4-D map over the [B][T][H][d] fp32 retention: boxes of 32 channels x 128 tokens, no
// swizzle, or (swz) with the 128-byte swizzle, so that a thread per token reading its row
// and a thread per channel reading a column both spread over the banks (al_swz).
inline bool make_tmap_alpha(CUtensorMap* m, const LinearProblem& p, bool swz = false) {
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
  cuuint64_t dims[4] = {(cuuint64_t)p.d, (cuuint64_t)p.T, (cuuint64_t)p.H, (cuuint64_t)p.B};
  cuuint64_t strides[3] = {(cuuint64_t)p.sT * 4, (cuuint64_t)p.sH * 4, (cuuint64_t)p.sB * 4};
  cuuint32_t box[4] = {32, (cuuint32_t)LT, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<float*>(p.alpha), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            swz ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D map over the bf16 C0 rows of the workspace: [rows][64], boxes of D rows, 128-byte
// swizzle (the MN-major B layout of the E = Qs C_0 product).
inline bool make_tmap_c0(CUtensorMap* m, void* base, long long rows, int d) {
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
  cuuint64_t dims[2] = {64, (cuuint64_t)rows};
  cuuint64_t strides[1] = {128};
  cuuint32_t box[2] = {64, (cuuint32_t)d};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t bwd_bytes(long long heads, long long nb, int d, LinCp* cp, __nv_bfloat16** dcb,
                 void* base);
template <int D>
cudaError_t states_t(const LinearProblem& lp, const void* dy, void* workspace, cudaStream_t s);

}  // namespace lintc
}  // namespace rel
