/*
 * relation.h -- C ABI of the GB300 (sm_103a) FlashRelation library.
 *
 * The library computes the exact causal Multi-Head Relation operator of
 * "Ask Self, Ask Others: Relation Is All You Need" (arxiv 2608.20172), forward and
 * backward, in tiled FlashRelation form: the T x T matrices U, R and F are never
 * written to memory.
 *
 * Per head, with p1 = Q (P1 after RoPE), p2 = K (P2 after RoPE) and I~ = V (the
 * information state after head mixing), rows i = 1..T (one-based):
 *   U_ij = p1_i . p2_j / sqrt(d_h)                           Eq. (relation-projections)
 *   S_i  = sigmoid(U_ii / tau_S),  E_ij = SiLU(U_ij)          Eq. (causal-relation)
 *   R_ii = S_i,  R_ij = E_ij - lambda log i (j < i),  R_ij = -inf (j > i)
 *   F_i  = Softmax(R_i),  Y_i = sum_{j<=i} F_ij I~_j          Eq. (relation-flow)
 * evaluated through the exact factorisation (Sec. 4.2 and Sec. 5.1):
 *   L^E_i = LSE_{j<i} E_ij (online scan), A_i = L^E_i - lambda log i,
 *   g_i = sigmoid(A_i - S_i), Y_i = (1 - g_i) I~_i + g_i Ibar_i, Ibar_i = sum pi^E_ij I~_j.
 * Row 1 has no history: g_1 = 0 and Y_1 = I~_1 (App. A.1.8).  Logarithms are natural.
 * lambda is one fp32 scalar per layer, shared by all heads (App. A.1.1); tau_S > 0
 * (the paper fixes tau_S = 2, Sec. 3.1) and carries no gradient.
 *
 * Conventions shared by every entry point
 *  - Tensors Q, K, V, O, dO, dQ, dK, dV are [B][T][H][d_h] with d_h contiguous and the
 *    element strides sB, sT, sH of relation_shape (so [B][H][T][d_h] works too).  All
 *    eight tensors use the same strides and dtype.  logZ is a dense fp32 [B][H][T].
 *  - Every pointer is a device pointer (cudaMalloc / cudaMallocAsync / managed).  The
 *    caller owns every buffer, including the backward workspace; the library allocates
 *    no memory and keeps no per-call state.
 *  - Calls are asynchronous on `stream` (NULL = the legacy default stream).
 *  - Argument errors are reported synchronously by the return value and nothing is
 *    launched.  A kernel whose pipeline wait exceeds its bound writes
 *    RELATION_ERR_TIMEOUT into *dev_status (a device int the caller zeroes and reads
 *    after synchronising; may be NULL) and returns without finishing its tile.
 *  - Supported: fp32 with d_h in {32, 64, 128} (CUDA-core kernels); bf16 with any d_h
 *    that is a multiple of 8 up to 128 (tcgen05 tensor-core kernels, zero-padded to 64
 *    or 128 inside; d_h 32, 64 and 128 also on the CUDA-core kernels).  Any T >= 1.
 *  - Alignment: every tensor pointer 16-byte aligned and sB, sT, sH multiples of
 *    16 bytes / element size; workspace 256-byte aligned.
 */
#ifndef RELATION_H
#define RELATION_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t / CUstream. */
typedef struct CUstream_st* relation_stream_t;

typedef enum relation_status {
  RELATION_OK = 0,
  RELATION_ERR_INVALID_ARG = 1, /* null pointer, bad size, non-finite lambda or tau_S   */
  RELATION_ERR_UNSUPPORTED = 2, /* d_h / dtype combination not built                     */
  RELATION_ERR_ALIGNMENT = 3,   /* pointer or stride alignment rule broken               */
  RELATION_ERR_WORKSPACE = 4,   /* workspace missing or smaller than the size query      */
  RELATION_ERR_CUDA = 5,        /* a CUDA runtime call failed (launch, attribute, ...)   */
  RELATION_ERR_TIMEOUT = 6      /* written to *dev_status by a kernel whose wait expired */
} relation_status;

typedef enum relation_dtype { RELATION_F32 = 0, RELATION_BF16 = 1 } relation_dtype;

typedef struct relation_shape {
  int B;        /* batch                                          */
  int T;        /* sequence length, >= 1                          */
  int H;        /* heads (MHR, Sec. 3.2)                           */
  int d_h;      /* head width                                     */
  long long sB; /* element stride between batches                 */
  long long sT; /* element stride between tokens                  */
  long long sH; /* element stride between heads; d_h is contiguous */
} relation_shape;

/*
 * Forward (Eqs. causal-relation, relation-flow; Sec. 5.1 and App. A.3).
 *   q, k, v : inputs P1, P2 (after RoPE) and I~ (after Givens mixing), dtype dt.
 *   o       : output Y, dtype dt, same layout.
 *   logz    : output fp32 [B][H][T], logZ_i = log sum_j exp(R_ij) = logaddexp(S_i, A_i)
 *             (logZ_1 = S_1).  This is the per-row statistic relation_bwd consumes.
 *   lambda  : count-calibration scalar lambda_l; tau_s: Self temperature (> 0).
 */
relation_status relation_fwd(const void* q, const void* k, const void* v, void* o, float* logz,
                             float lambda, float tau_s, relation_shape shp, relation_dtype dt,
                             int* dev_status, relation_stream_t stream);

/* Kernel family selection for the *_ex entry points.  AUTO takes the tcgen05
 * tensor-core kernels where they exist (bf16, d_h a multiple of 8 up to 128) and the
 * CUDA-core (SIMT) kernels otherwise; TCGEN05 returns RELATION_ERR_UNSUPPORTED where they
 * do not exist. */
typedef enum relation_kernel {
  RELATION_KERNEL_AUTO = 0,
  RELATION_KERNEL_SIMT = 1,
  RELATION_KERNEL_TCGEN05 = 2
} relation_kernel;

/* relation_fwd with an explicit kernel family (relation_fwd == relation_fwd_ex(..., AUTO)). */
relation_status relation_fwd_ex(const void* q, const void* k, const void* v, void* o, float* logz,
                                float lambda, float tau_s, relation_shape shp, relation_dtype dt,
                                relation_kernel kernel, int* dev_status, relation_stream_t stream);

/*
 * relation_fwd_ex with one more output, the Self flow of every row:
 *   self_flow [B][H][T] fp32 : F_ii = exp(R_ii - logZ_i) = sigmoid(S_i - A_i) = 1 - g_i,
 * the share of row i's normalised flow F that stays on the Self relation (Sec. 4.2, the
 * Self-Exchange factorisation; its complement g_i is the Exchange share).  This is the
 * per-row quantity behind the paper's "Self flow" and "Self / Exchange" structural
 * diagnostics (App. B.4, B.5); averaging it is left to the caller.  Row 1 has no history: F_11 = 1.  self_flow may be null (then this is
 * relation_fwd_ex); otherwise it must be 16-byte aligned.  Y and logz are identical to
 * relation_fwd_ex's.
 */
relation_status relation_fwd_flow(const void* q, const void* k, const void* v, void* o,
                                  float* logz, float* self_flow, float lambda, float tau_s,
                                  relation_shape shp, relation_dtype dt, relation_kernel kernel,
                                  int* dev_status, relation_stream_t stream);

/*
 * Linear Relation forward (Sec. 5.2, Eq. (decayed-relation-state); App. A.4): the
 * recurrent Exchange form, per head with the d_h x d_h state C_0 = 0,
 *   S_t = sigmoid(p1_t . p2_t / (tau_S sqrt d_h)),  ^p = p / |p|
 *   C^- = Diag(alpha_t) C_{t-1},  E_t = S_t (C^-)^T ^p1_t,  Y_t = I~_t + E_t,
 *   C_t = C^- + S_t ^p2_t I~_t^T.
 *   p1, p2, v : [B][T][H][d_h] relation coordinates (after RoPE) and information, in dt.
 *   alpha     : [B][T][H][d_h] fp32 channel-wise retention in (0, 1] (the KDA-style
 *               parameterisation of Eq. (retention-vector) is upstream), with the same
 *               element strides as p1.
 *   y         : [B][T][H][d_h] output in dt, same strides.
 * fp32 or bf16 with d_h in {32, 64, 128} (other widths: RELATION_ERR_UNSUPPORTED); the state is
 * kept in fp32.  Element strides sB, sT, sH must be multiples of 4 and every pointer
 * 16-byte aligned (else RELATION_ERR_ALIGNMENT).  A zero p1 or p2 row is outside the
 * operator's domain.  Asynchronous on `stream`; nothing is allocated.
 */
relation_status relation_linear_fwd(const void* p1, const void* p2, const void* v,
                                   const float* alpha, void* y, float tau_s, relation_shape shp,
                                   relation_dtype dt, int* dev_status, relation_stream_t stream);

/*
 * relation_linear_fwd with a choice of kernel family (relation_linear_fwd uses AUTO):
 *   RELATION_KERNEL_SIMT    the token-sequential recurrence on CUDA cores (every dtype and
 *                           width above; the state and all products in fp32).
 *   RELATION_KERNEL_TCGEN05 the chunked form on the tensor cores: blocks of 128 tokens, the
 *                           within-block pairs and the state's read and update as tcgen05
 *                           products with bf16 operands and fp32 accumulation, the fp32 state
 *                           in tensor memory.  bf16 with d_h 64 or 128 only, element strides
 *                           multiples of 8 (else RELATION_ERR_UNSUPPORTED or
 *                           RELATION_ERR_ALIGNMENT, nothing launched).  The retention ratios
 *                           a_t / a_j inside a block are split at its midpoint, so a factor
 *                           covers at most 64 tokens of decay: a channel whose retention
 *                           product over 64 consecutive tokens of one block falls below 2^-120
 *                           has its factor clamped, the result is then not exact, and
 *                           RELATION_ERR_UNSUPPORTED is written to *dev_status (non-null) once
 *                           the call completes.
 *   RELATION_KERNEL_AUTO    the chunked kernel where it applies, else the recurrence.
 */
relation_status relation_linear_fwd_ex(const void* p1, const void* p2, const void* v,
                                      const float* alpha, void* y, float tau_s,
                                      relation_shape shp, relation_dtype dt,
                                      relation_kernel kernel, int* dev_status,
                                      relation_stream_t stream);

/*
 * relation_linear_fwd with a caller workspace, for long sequences.  The chunked kernel walks
 * a head's 128-token blocks in order, one CTA per (head, 64 information columns), so a call
 * with fewer such pairs than the GPU has SMs leaves SMs idle.  With a workspace the blocks
 * run in parallel instead: every block's state contribution (its decayed sum of k' I~^T and
 * its decay, fp32), then a scan of the state over the blocks, then every block's output from
 * the state it starts from (stored in bf16 between the passes; three launches).
 *   workspace : device scratch of relation_linear_fwd_workspace_size(shp, dt) bytes
 *               (B H (d_h / 64) ceil(T / 128) d_h rows of 64 + 1 fp32, and
 *               B H (d_h / 64) (ceil(T / 128) + 1) d_h rows of 64 bf16),
 *               16-byte aligned, or RELATION_ERR_WORKSPACE / RELATION_ERR_ALIGNMENT with
 *               nothing launched.
 * The chunk-parallel form runs when B H (d_h / 64) is below half the device's SM count, the
 * sequential chunked kernel otherwise (same results up to rounding).  Requests the chunked
 * kernel does not serve (workspace size 0: fp32, d_h other than 64 and 128, strides not
 * multiples of 8) go to relation_linear_fwd_ex(..., RELATION_KERNEL_AUTO, ...) and ignore the
 * workspace.  Other arguments, results and the decay-range report are those of
 * relation_linear_fwd_ex with RELATION_KERNEL_TCGEN05.
 */
size_t relation_linear_fwd_workspace_size(relation_shape shp, relation_dtype dt);
relation_status relation_linear_fwd_ws(const void* p1, const void* p2, const void* v,
                                      const float* alpha, void* y, float tau_s,
                                      relation_shape shp, relation_dtype dt, void* workspace,
                                      size_t ws_bytes, int* dev_status,
                                      relation_stream_t stream);

/*
 * Linear Relation backward: the reverse-mode derivative of the recurrence above (the paper
 * writes out the forward only), given dy = dL/dY:
 *   dp1, dp2, dv : [B][T][H][d_h] in dt, with the inputs' strides (overwritten);
 *   dalpha       : [B][T][H][d_h] fp32 with alpha's strides (overwritten);
 *   workspace    : device scratch of relation_linear_bwd_workspace_size(shp, dt) bytes,
 *                  the size relation_linear_bwd_ex_workspace_size gives for
 *                  RELATION_KERNEL_AUTO (16-byte aligned).
 * Same dtypes and widths as relation_linear_fwd; asynchronous on `stream`.  Equals
 * relation_linear_bwd_ex(..., RELATION_KERNEL_AUTO, ...).
 */
size_t relation_linear_bwd_workspace_size(relation_shape shp, relation_dtype dt);
relation_status relation_linear_bwd(const void* p1, const void* p2, const void* v,
                                   const float* alpha, const void* dy, void* dp1, void* dp2,
                                   void* dv, float* dalpha, float tau_s, relation_shape shp,
                                   relation_dtype dt, void* workspace, size_t ws_bytes,
                                   int* dev_status, relation_stream_t stream);

/*
 * relation_linear_bwd with the kernel family chosen (relation_kernel, as for the forward):
 *   RELATION_KERNEL_SIMT    reverse mode through the token recurrence on CUDA cores (every
 *                           dtype and width of relation_linear_fwd).  Workspace: state
 *                           checkpoints every 8 tokens plus fp32 partial row sums of the
 *                           state's column splits, B H (ceil(T / 8) d_h^2 + (d_h / 32) T 3 d_h)
 *                           fp32.
 *   RELATION_KERNEL_TCGEN05 reverse mode through the 128-token blocks of the chunked
 *                           forward, every block in parallel: the states entering every block
 *                           (a forward state pass), the state's adjoint leaving every block
 *                           (dC(b - 1) = Diag(a_L(b)) dC(b) + Qs_b^T dY_b, a reverse pass),
 *                           then per block the gradients as tcgen05 products with bf16
 *                           operands and fp32 accumulation (five launches).  bf16 with d_h = 64,
 *                           element strides multiples of 8 (else RELATION_ERR_UNSUPPORTED or
 *                           RELATION_ERR_ALIGNMENT, nothing launched).  Workspace, in
 *                           256-byte-aligned parts, with n = ceil(T / 128): B H n 64 rows of 64
 *                           fp32, B H n 64 fp32, B H (n + 1) 64 rows of 64 bf16 (the states,
 *                           the final one last) and B H n 64 rows of 64 bf16 (the adjoints).
 *                           The decay-range clamp and its report are the chunked forward's.
 *   RELATION_KERNEL_AUTO    the chunked kernel where it applies, else the recurrence.
 * workspace is 16-byte aligned and holds relation_linear_bwd_ex_workspace_size(shp, dt,
 * kernel) bytes (0: the family does not serve the request), else RELATION_ERR_WORKSPACE /
 * RELATION_ERR_ALIGNMENT with nothing launched.  Other arguments as relation_linear_bwd.
 */
size_t relation_linear_bwd_ex_workspace_size(relation_shape shp, relation_dtype dt,
                                             relation_kernel kernel);
relation_status relation_linear_bwd_ex(const void* p1, const void* p2, const void* v,
                                      const float* alpha, const void* dy, void* dp1, void* dp2,
                                      void* dv, float* dalpha, float tau_s, relation_shape shp,
                                      relation_dtype dt, relation_kernel kernel, void* workspace,
                                      size_t ws_bytes, int* dev_status, relation_stream_t stream);

/*
 * Decoding: the forward row of one new token per sequence, against a key/value cache.
 *   q        [B][H][d_h] queries of the new tokens, element strides q_sB, q_sH (d_h
 *            contiguous); o (output Y) has the same layout.
 *   k_cache, v_cache : [B][T][H][d_h] with the strides of `cache` (T = cache capacity).
 *   lengths  device int[B]: rows of sequence b in the cache, 1 <= len_b <= T; row
 *            len_b - 1 holds the new token's key and value, and len_b is its one-based
 *            position i in ln(i).
 *   logz     [B][H] fp32 output: log of the new row's normaliser.
 *   workspace, ws_bytes : device scratch of relation_decode_workspace_size(cache, dt).
 * Y and logz equal row len_b - 1 of relation_fwd over the first len_b cache rows (the
 * Self-Exchange row of Sec. 3.1 in the factorised form of Sec. 4.2): Exchange over the
 * len_b - 1 history rows, Self with the token's own key.  bf16 or fp32 with any 1 <= d_h <= 128.
 * A length outside [1, T] is not read: the heads of that sequence are skipped and
 * dev_status (if given) receives RELATION_ERR_INVALID_ARG.  Asynchronous on `stream`.
 */
size_t relation_decode_workspace_size(relation_shape cache, relation_dtype dt);
relation_status relation_decode(const void* q, const void* k_cache, const void* v_cache,
                                const int* lengths, void* o, float* logz, float lambda,
                                float tau_s, relation_shape cache, long long q_sB, long long q_sH,
                                relation_dtype dt, void* workspace, size_t ws_bytes,
                                int* dev_status, relation_stream_t stream);

/*
 * Context parallelism (sequence sharding) of the forward.  The Exchange summary of a query
 * row over a set of history keys is (m, l, z): l = sum_j exp(E_ij - m) and
 * z = sum_j exp(E_ij - m) I~_j over those keys, for any log-scale m (here an upper bound of
 * their max E); summaries over disjoint key sets merge associatively (App. A.3, the online
 * update of the scan), and the epilogue of App. A.3.3-A.3.5 needs only the merged summary,
 * the row's own q_i, k_i (Self) and v_i, and its position i.  A sequence split into shards
 * of consecutive tokens is thus computed shard by shard:
 *   relation_fwd_state(causal = 1) over the shard's own tokens, then for every earlier
 *   shard relation_fwd_state(causal = 0) of the shard's queries against that shard's keys
 *   and relation_state_merge into the first, then relation_state_finish with pos0 = the
 *   shard's first position -- Y and logZ equal relation_fwd over the whole sequence up to
 *   rounding.
 * Summary layout (dense, fp32, caller-owned): m, l [B][H][T_q], z [B][H][T_q][d_h].
 *
 * relation_fwd_state: the summary of every row of q ([B][T_q][H][d_h], strides of shp_q)
 *   over the keys of k, v ([B][T_k][H][d_h], strides of shp_kv; B, H, d_h as shp_q):
 *   causal = 1: k, v are the queries' own tokens (T_k = T_q), row i takes keys j < i (Self
 *   excluded; row 0's summary is empty: m = -inf, l = 0, z = 0); causal = 0: every one of
 *   the T_k keys precedes every query.  bf16 with d_h a multiple of 8 up to 128 (the
 *   tensor-core forward's tiles; otherwise RELATION_ERR_UNSUPPORTED).
 * relation_state_merge: (m, l, z) <- merge of (m, l, z) and (m2, l2, z2), rows of
 *   shp.B, shp.H, shp.T (strides ignored), d_h <= 128 a multiple of 4.
 * relation_state_finish: Y (o, [B][T][H][d_h] with q's strides, dt) and logZ ([B][H][T]
 *   fp32) of the rows of q, k, v from their summaries; row r sits at one-based position
 *   pos0 + r + 1 of the sequence (the ln i of the count term); self_flow (optional) gets
 *   F_ii.  bf16 or fp32, d_h <= 128 a multiple of 4.
 * All three are asynchronous on `stream`; nothing is launched on an argument error.
 */
relation_status relation_fwd_state(const void* q, const void* k, const void* v, float* m,
                                   float* l, float* z, relation_shape shp_q,
                                   relation_shape shp_kv, int causal, relation_dtype dt,
                                   int* dev_status, relation_stream_t stream);
relation_status relation_state_merge(float* m, float* l, float* z, const float* m2,
                                     const float* l2, const float* z2, relation_shape shp,
                                     relation_stream_t stream);
relation_status relation_state_finish(const void* q, const void* k, const void* v,
                                      const float* m, const float* l, const float* z, void* o,
                                      float* logz, float* self_flow, float lambda, float tau_s,
                                      long long pos0, relation_shape shp, relation_dtype dt,
                                      relation_stream_t stream);

/*
 * The paper layer's transforms around the operator (Sec. 3.1-3.2, Eq. (givens-rotation),
 * App. A.2.2, App. B.3), producing the operator's inputs from the projected states:
 *   q = RoPE(p1), k = RoPE(p2): full-head rotary embedding, channel pairs (2c, 2c+1)
 *       of the row at position m (zero-based, restarting at every sequence) turned by
 *       m * rope_base^(-2c/d_h) (the paper's base is 1e4);
 *   v = Givens(info): head pairs (a, b) mixed on every channel with angle theta[k],
 *       v_a = cos info_a - sin info_b,  v_b = sin info_a + cos info_b;
 *       pairing 0: (0,1), (2,3), ..., (H-2,H-1); pairing 1: (1,2), ..., (H-1,0) (the
 *       paper's alternating sets M_A and M_B, zero-based).
 *   p1, p2, info, q, k, v : [B][T][H][d_h] in dt with the strides of `shp`; each output
 *       may alias its input (q = p1, k = p2, v = info).
 *   theta : device float[H/2], fp32.
 * H even, d_h a multiple of 8 up to 256, H/2 <= 128; fp32 or bf16 (rotations in fp32; the
 * RoPE angles are reduced modulo 2 pi in fp64).  Other shapes: RELATION_ERR_UNSUPPORTED.
 * Asynchronous on `stream`; nothing is allocated.
 */
relation_status relation_layer_prep(const void* p1, const void* p2, const void* info,
                                    const float* theta, int pairing, float rope_base, void* q,
                                    void* k, void* v, relation_shape shp, relation_dtype dt,
                                    relation_stream_t stream);

/*
 * Gradient of relation_layer_prep: from the operator's dq, dk, dv (as relation_bwd
 * returns them) and the forward's info and theta,
 *   dp1 = RoPE^T(dq), dp2 = RoPE^T(dk), dinfo = Givens^T(dv) (each may alias its input),
 *   dtheta : device float[H/2], dtheta_k = sum over b, t, channels of
 *            dv_a (-sin info_a - cos info_b) + dv_b (cos info_a - sin info_b)
 *            (overwritten; summed in a fixed order, deterministic);
 *   workspace : device scratch of relation_layer_grad_workspace_size(shp, dt) bytes.
 * Same shapes and dtypes as relation_layer_prep; asynchronous on `stream`.
 */
size_t relation_layer_grad_workspace_size(relation_shape shp, relation_dtype dt);
relation_status relation_layer_grad(const void* dq, const void* dk, const void* dv,
                                    const void* info, const float* theta, int pairing,
                                    float rope_base, void* dp1, void* dp2, void* dinfo,
                                    float* dtheta, relation_shape shp, relation_dtype dt,
                                    void* workspace, size_t ws_bytes, relation_stream_t stream);

/* Bytes of device workspace relation_bwd needs for this shape and dtype (0 on a bad
 * shape).  The content of the workspace need not be initialised. */
size_t relation_bwd_workspace_size(relation_shape shp, relation_dtype dt);

/*
 * Backward (App. A.1.7), recomputing the tiles from logz.
 *   q, k, v, o, dout, logz : the forward's inputs, its output Y, dL/dY and its logz.
 *   dq, dk, dv             : outputs dL/dP1, dL/dP2, dL/dI~ (overwritten, not accumulated).
 *   dlambda                : output, one device float, dL/dlambda summed over B, H and T
 *                            (lambda is shared by the heads).  Overwritten.
 *   workspace, ws_bytes    : device scratch of at least relation_bwd_workspace_size().
 * The gradient follows the generic softmax form dR_ij = F_ij (H_ij - D_i) with
 * H_ij = dO_i . I~_j and D_i = dO_i . Y_i, chained through sigma' (Self, with 1/tau_S)
 * and SiLU' (Exchange).  dlambda = -sum_i log i sum_{j<i} dR_ij = sum_i log i dR_ii,
 * because every row of dR sums to zero.
 */
relation_status relation_bwd(const void* q, const void* k, const void* v, const void* o,
                             const void* dout, const float* logz, void* dq, void* dk, void* dv,
                             float* dlambda, float lambda, float tau_s, relation_shape shp,
                             relation_dtype dt, void* workspace, size_t ws_bytes,
                             int* dev_status, relation_stream_t stream);

/* relation_bwd with an explicit kernel family (relation_bwd == relation_bwd_ex(..., AUTO)). */
relation_status relation_bwd_ex(const void* q, const void* k, const void* v, const void* o,
                                const void* dout, const float* logz, void* dq, void* dk, void* dv,
                                float* dlambda, float lambda, float tau_s, relation_shape shp,
                                relation_dtype dt, void* workspace, size_t ws_bytes,
                                relation_kernel kernel, int* dev_status, relation_stream_t stream);

/* Number of kernel launches one relation_fwd_ex (backward = 0) or relation_bwd_ex
 * (backward != 0) call makes for this dtype, head width and kernel request; 0 when the
 * request is not supported.  Host-only query. */
int relation_launch_count(relation_dtype dt, int d_h, relation_kernel kernel, int backward);

/* The backward as three stages, each launched only when its bit is set in `stages`:
 *   RELATION_BWD_PREPARE  per-row pass: D_i = dO_i . Y_i, the Self quantities and the
 *                         per-query scalars the tile stage reads (into the workspace)
 *   RELATION_BWD_TILES    the causal tile loop producing dK, dV and the dQ accumulator
 *   RELATION_BWD_FINALIZE dQ in the output dtype and the dlambda reduction
 * Running the three in order on one stream (stages = RELATION_BWD_ALL) is relation_bwd_ex.
 * The stages communicate through the workspace only; a stage assumes the earlier ones ran
 * on the same arguments and workspace. */
enum { RELATION_BWD_PREPARE = 1, RELATION_BWD_TILES = 2, RELATION_BWD_FINALIZE = 4,
       RELATION_BWD_ALL = 7 };
relation_status relation_bwd_stages(const void* q, const void* k, const void* v, const void* o,
                                    const void* dout, const float* logz, void* dq, void* dk,
                                    void* dv, float* dlambda, float lambda, float tau_s,
                                    relation_shape shp, relation_dtype dt, void* workspace,
                                    size_t ws_bytes, relation_kernel kernel, unsigned stages,
                                    int* dev_status, relation_stream_t stream);

/*
 * relation_bwd without a caller workspace, for callers that cannot allocate device memory
 * (code inside a runtime that owns the device memory budget through its own allocator, or
 * on a path where an allocation could fail or synchronise the device).  The paper has no
 * counterpart: this is a deployment convenience.
 *
 * The scratch is a fixed device array of RELATION_STATIC_SCRATCH_BYTES inside the library,
 * held on every GPU that loads the library until the process exits.  Shapes whose
 * relation_bwd_workspace_size() exceeds it are rejected with RELATION_ERR_WORKSPACE and
 * nothing is launched.  The operands must be on the device current on the calling thread
 * (that device's copy of the array is used); a q that is not device memory of that device
 * is rejected with RELATION_ERR_INVALID_ARG and nothing is launched.  Each call looks up
 * the array's address on the current device.  Under CUDA's lazy module loading, the first
 * call on a device (or the library's first launch there) loads the module and so commits
 * the RELATION_STATIC_SCRATCH_BYTES at that moment: a caller whose allocator owns the
 * memory budget should make one call during set-up, before any stream capture (and again
 * after a device reset).  No call allocates memory otherwise.  Every call shares the one
 * array: calls that overlap on the GPU race on it and must be serialised by the caller.
 * Arguments and results are otherwise those of relation_bwd_ex.
 */
#define RELATION_STATIC_SCRATCH_BYTES (64u << 20)
relation_status relation_bwd_static(const void* q, const void* k, const void* v, const void* o,
                                    const void* dout, const float* logz, void* dq, void* dk,
                                    void* dv, float* dlambda, float lambda, float tau_s,
                                    relation_shape shp, relation_dtype dt, relation_kernel kernel,
                                    int* dev_status, relation_stream_t stream);

/* Human-readable name of a status code (static string, never NULL). */
const char* relation_status_string(relation_status s);

/* When a call returned RELATION_ERR_CUDA: the CUDA error string of the failing CUDA call
 * made by the calling thread inside the library ("no error" otherwise).  Static string. */
const char* relation_last_cuda_error(void);

/* Library ABI version, (major << 16) | minor. */
int relation_version(void);

/*
 * Self-test of the bounded pipeline wait used by every tensor-core kernel: launches
 * one tiny kernel that waits on an mbarrier nothing will ever complete, with a bound of
 * about `timeout_us` microseconds (1..100000).  On expiry the kernel writes
 * RELATION_ERR_TIMEOUT into *dev_status and returns; the context stays usable.
 * The paper has no counterpart: this exists to test failure detection.
 */
relation_status relation_selftest_wait_timeout(int* dev_status, int timeout_us,
                                               relation_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* RELATION_H */
