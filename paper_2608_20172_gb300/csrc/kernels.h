// kernels.h -- internal launch interface between the C ABI layer and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>

#include "relation.h"

namespace rel {

// Everything a kernel launch needs; pointers are device pointers.
struct Problem {
  // tensors ([B][T][H][d] with element strides sB, sT, sH)
  const void* q;
  const void* k;
  const void* v;
  const void* o;     // forward output (read by the backward)
  const void* dout;  // dL/dY
  void* out;         // forward: Y
  void* dq;
  void* dk;
  void* dv;
  float* logz;         // forward output [B][H][T]
  float* fself;        // optional forward output [B][H][T]: the Self flow F_ii (may be null)
  const float* logz_in;  // backward input [B][H][T]
  float* dlambda;      // backward output (one float)
  int* dev_status;
  // scalars
  float lambda;
  float tau_s;
  float inv_sqrt_d;
  int B, T, H, d;
  long long sB, sT, sH;
  relation_dtype dtype;
};

// The Exchange summary of a forward over part of the keys (context parallelism): per query
// row the log-scale m (natural log), the sum l = sum_j exp(E_ij - m) and the unnormalised
// z = sum_j exp(E_ij - m) v_j over the keys visited; Self is never part of it.
struct StateArgs {
  int causal;                    // 1: keys = the queries' own tokens (j < i); 0: all keys
  int Tk;                        // keys (causal: = T)
  long long k_sB, k_sT, k_sH;    // element strides of k and v (causal: the queries')
  float* m;                      // [B][H][T]
  float* l;                      // [B][H][T]
  float* z;                      // [B][H][T][d] (d real columns)
};

// Context parallelism (relation_cp.cu): merge (m2, l2, z2) into (m, l, z) over `rows` rows
// of d <= 128 columns; the epilogue of p's rows from their summaries, the first row at
// zero-based position pos0 of the sequence (reads p.q, p.k, p.v; writes p.out, p.logz and,
// if set, p.fself).
cudaError_t launch_state_merge(float* m, float* l, float* z, const float* m2, const float* l2,
                               const float* z2, long long rows, int d, cudaStream_t s);
cudaError_t launch_state_finish(const Problem& p, const float* m, const float* l, const float* z,
                                long long pos0, cudaStream_t s);

// Backward workspace carved out of the caller's buffer (all fp32, 256-byte aligned).
struct BwdWorkspace {
  float* dq_acc;     // [B][H][T_pad][d_pad] 2 sqrt(d) dL/dP1 in fp32, T_pad = T rounded up to
                     //   128, d_pad = d rounded up to 64
                     //   (tensor-core path: zeroed by its row pass, then summed by TMA reduce)
  int t_pad;
  float* D;          // [B][H][T]     D_i = dO_i . Y_i
  float* F_self;     // [B][H][T]     F_ii = exp(S_i - logZ_i)
  float* dS_self;    // [B][H][T]     dL/du_ii, u = U_ii (scaled evidence)
  float* wl;         // [B][H][T]     log i F_ii (dlambda weight of row i's Exchange pairs)
  float* stats;      // [B][H][T_pad/128][3][128] per-query scalars of the tensor-core backward
  // dlambda partials: [n_pre_blocks] from the row pre-pass (the Self terms; the SIMT pass
  // fills the first ceil(rows / 8), the tensor-core pass the first T_pad B H / 32), then
  // [n_main_slots] from the Exchange tile kernel (one per CTA).
  float* dlam_part;
  int n_pre_blocks;
  int n_main_slots;  // capacity reserved for the tile kernel's CTAs
};

size_t bwd_workspace_bytes(int B, int H, int T, int d);
BwdWorkspace carve_workspace(void* base, int B, int H, int T, int d);

namespace simt {
bool supports(relation_dtype dt, int d);
cudaError_t launch_fwd(const Problem& p, cudaStream_t s);
cudaError_t launch_bwd(const Problem& p, const BwdWorkspace& ws, cudaStream_t s);
int main_ctas(const Problem& p);  // tile-kernel CTAs writing a dlambda partial
}  // namespace simt

namespace bwd_common {
// Per-row Self part of the CUDA-core backward (D_i, F_ii, dS_ii and dlambda partials).
cudaError_t launch_pre(const Problem& p, const BwdWorkspace& ws, cudaStream_t s);
// Deterministic dlambda reduction of the pre-pass partials and the first n_main tile-kernel
// partials.
cudaError_t launch_dlambda(const Problem& p, const BwdWorkspace& ws, int n_main, cudaStream_t s);
}  // namespace bwd_common

namespace tc {
// Number of head groups of the tile kernels' work order (grouped_unit in common.cuh):
// every group holds at least ceil(2.5 slots / (n_t + 1)) heads, so that one group's work
// per resident CTA slot covers its heaviest unit (n_t tiles) with margin.  `slots` = CTAs
// resident at once over the whole GPU.
inline int head_groups(int n_t, int BH, int slots) {
  long long g = (5LL * slots + 2LL * (n_t + 1) - 1) / (2LL * (n_t + 1));
  if (g < 1) g = 1;
  const long long n = BH / g;
  return n < 1 ? 1 : (int)n;
}
bool supports(relation_dtype dt, int d);      // forward
bool supports_bwd(relation_dtype dt, int d);  // backward
cudaError_t launch_fwd(const Problem& p, cudaStream_t s);
// The forward's scan without its epilogue: the Exchange summary of every query row over
// the keys of st (causal: the queries' own earlier tokens; else every key of k, v), written
// to st.m, st.l, st.z (relation_tc_fwd.cu).
cudaError_t launch_fwd_state(const Problem& p, const StateArgs& st, cudaStream_t s);
// Backward stages (bit 1: row pass, 2: tile kernel, 4: finalisation).
cudaError_t launch_bwd(const Problem& p, const BwdWorkspace& ws, unsigned stages, cudaStream_t s);
int bwd_launches();  // launches made by launch_bwd with every stage
int main_ctas(const Problem& p);
}  // namespace tc

// Decoding: one new token per sequence against a key/value cache (relation_decode.cu).
struct DecodeProblem {
  const void* q;        // [B][H][d] queries of the new tokens (element strides qsB, qsH)
  const void* k;        // caches [B][T][H][d] (element strides sB, sT, sH); row len_b - 1 of
  const void* v;        //   sequence b is the new token
  const int* lengths;   // device [B]: cached rows per sequence, 1 <= len_b <= T
  void* out;            // [B][H][d] like q
  float* logz;          // [B][H]
  int* dev_status;      // nullable: RELATION_ERR_INVALID_ARG for a length outside [1, T]
  float lambda, tau_s, inv_sqrt_d;
  int B, T, H, d;
  long long sB, sT, sH, qsB, qsH;
  relation_dtype dtype;
};
// Linear Relation (relation_linear.cu).
struct LinearProblem {
  const void* p1;       // [B][T][H][d] relation coordinates after RoPE (strides sB, sT, sH)
  const void* p2;
  const void* v;        // information I~
  const float* alpha;   // retention in (0, 1], fp32, same shape and element strides
  void* y;              // forward output
  const void* dy;       // backward input dL/dY
  void* dp1;            // backward outputs (input dtype), dalpha fp32
  void* dp2;
  void* dv;
  float* dalpha;
  void* workspace;      // backward scratch
  int* dev_status;
  float tau_s;
  int B, T, H, d;
  long long sB, sT, sH;
  relation_dtype dtype;
};
bool linear_supports(relation_dtype dt, int d);
cudaError_t launch_linear_fwd(const LinearProblem& p, cudaStream_t s);
// Chunked tensor-core forward (relation_linear_tc.cu): bf16, d_h 64 or 128, element
// strides multiples of 8.
// workspace == nullptr: one CTA per (head, 64 columns) walks the blocks in order;
// otherwise the chunk-parallel form (every block's state contribution in parallel, a scan
// of the state over the blocks, every block's output in parallel) in that workspace of
// linear_tc_workspace_bytes(p) bytes.
bool linear_tc_supports(const LinearProblem& p);
size_t linear_tc_workspace_bytes(const LinearProblem& p);
cudaError_t launch_linear_tc_fwd(const LinearProblem& p, void* workspace, cudaStream_t s);
// Chunked tensor-core backward (relation_linear_tc_bwd.cu): bf16, d_h 64, element strides
// multiples of 8; p.workspace holds linear_tc_bwd_workspace_bytes(p) bytes (the forward's
// block states and the state's adjoints, bf16).
bool linear_tc_bwd_supports(const LinearProblem& p);
size_t linear_tc_bwd_workspace_bytes(const LinearProblem& p);
cudaError_t launch_linear_tc_bwd(const LinearProblem& p, cudaStream_t s);
size_t linear_bwd_workspace_bytes(int B, int H, int T, int d);
cudaError_t launch_linear_bwd(const LinearProblem& p, cudaStream_t s);

// The layer's transforms around the operator (RoPE of P1, P2; Givens mixing of the
// information states) and their gradients.  prep: in1, in2, in3 = P1, P2, I and out1,
// out2, out3 = Q, K, V.  grad: in1, in2, in3 = dQ, dK, dV, in4 = I and out1, out2, out3 =
// dP1, dP2, dI, with dtheta [H/2] (fp32) and dtheta_part the per-CTA partials.
struct LayerProblem {
  const void* in1;
  const void* in2;
  const void* in3;
  const void* in4;
  void* out1;
  void* out2;
  void* out3;
  const float* theta;   // [H/2] Givens angles, fp32, device
  float* dtheta;        // [H/2], grad only
  float* dtheta_part;   // grad only: caller workspace
  int pairing;          // 0: (0,1), (2,3), ...; 1: (1,2), ..., (H-1,0)
  float rope_base;
  int B, T, H, d;
  long long sB, sT, sH;
  relation_dtype dtype;
};
bool layer_supports(relation_dtype dt, int d, int H);
size_t layer_grad_workspace_bytes(int B, int T, int H);
cudaError_t launch_layer_prep(const LayerProblem& p, cudaStream_t s);
cudaError_t launch_layer_grad(const LayerProblem& p, cudaStream_t s);

int decode_chunks(int t_max);
size_t decode_workspace_bytes(int B, int H, int t_max);
cudaError_t launch_decode(const DecodeProblem& p, void* workspace, cudaStream_t s);

cudaError_t launch_selftest_wait(int* dev_status, int timeout_us, cudaStream_t s);

// Where the last failing CUDA step of this thread happened (reported by
// relation_last_cuda_error); launchers set it before returning an error.
void note_failure(const char* where);

}  // namespace rel
