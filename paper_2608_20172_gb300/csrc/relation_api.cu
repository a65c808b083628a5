// relation_api.cu -- the C ABI of librelation (declared in include/relation.h).
//
// Host code only: argument validation (nothing is launched on an error), selection of
// the kernel family, workspace carving and launches on the caller's stream.  The
// library allocates no device memory.
#include <math.h>
#include <stdint.h>
#include <stdio.h>

#include "kernels.h"
#include "relation.h"

namespace {

using rel::Problem;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t elem_size(relation_dtype dt) { return dt == RELATION_F32 ? 4 : 2; }

relation_status check_shape(const relation_shape& s, relation_dtype dt) {
  if (dt != RELATION_F32 && dt != RELATION_BF16) return RELATION_ERR_INVALID_ARG;
  if (s.B < 1 || s.T < 1 || s.H < 1 || s.d_h < 1) return RELATION_ERR_INVALID_ARG;
  if ((long long)s.B * s.H > 65535) return RELATION_ERR_UNSUPPORTED;  // grid.y limit
  if (s.sB < 1 || s.sT < 1 || s.sH < 1) return RELATION_ERR_INVALID_ARG;
  if (!rel::simt::supports(dt, s.d_h) && !rel::tc::supports(dt, s.d_h))
    return RELATION_ERR_UNSUPPORTED;
  const long long vec = 16 / (long long)elem_size(dt);
  if (s.sB % vec || s.sT % vec || s.sH % vec) return RELATION_ERR_ALIGNMENT;
  return RELATION_OK;
}

relation_status check_scalars(float lambda, float tau_s) {
  if (!isfinite(lambda) || !isfinite(tau_s) || !(tau_s > 0.0f)) return RELATION_ERR_INVALID_ARG;
  return RELATION_OK;
}

relation_status check_ptrs(std::initializer_list<const void*> ptrs) {
  for (const void* p : ptrs)
    if (!p) return RELATION_ERR_INVALID_ARG;
  for (const void* p : ptrs)
    if (!aligned16(p)) return RELATION_ERR_ALIGNMENT;
  return RELATION_OK;
}

// Family that will run: 1 = SIMT, 2 = tcgen05; 0 when the request cannot be served.
int pick_family(relation_kernel kernel, relation_dtype dt, int d, bool backward) {
  const bool tc = backward ? rel::tc::supports_bwd(dt, d) : rel::tc::supports(dt, d);
  const bool simt = rel::simt::supports(dt, d);
  switch (kernel) {
    case RELATION_KERNEL_AUTO: return tc ? 2 : (simt ? 1 : 0);
    case RELATION_KERNEL_SIMT: return simt ? 1 : 0;
    case RELATION_KERNEL_TCGEN05: return tc ? 2 : 0;
  }
  return 0;
}

Problem make_problem(relation_shape s, relation_dtype dt, float lambda, float tau_s,
                     int* dev_status) {
  Problem p{};
  p.lambda = lambda;
  p.tau_s = tau_s;
  p.inv_sqrt_d = 1.0f / sqrtf((float)s.d_h);
  p.B = s.B; p.T = s.T; p.H = s.H; p.d = s.d_h;
  p.sB = s.sB; p.sT = s.sT; p.sH = s.sH;
  p.dtype = dt;
  p.dev_status = dev_status;
  return p;
}

thread_local cudaError_t g_last_cuda_error = cudaSuccess;
thread_local const char* g_last_where = "";
thread_local char g_last_message[256];

relation_status from_cuda(cudaError_t e) {
  if (e == cudaSuccess) return RELATION_OK;
  if (e == cudaErrorInvalidValue && !g_last_where[0]) g_last_where = "launch";
  g_last_cuda_error = e;
  return RELATION_ERR_CUDA;
}

}  // namespace

namespace rel {
void note_failure(const char* where) { g_last_where = where; }
}  // namespace rel

extern "C" {

relation_status relation_fwd_flow(const void* q, const void* k, const void* v, void* o,
                                  float* logz, float* self_flow, float lambda, float tau_s,
                                  relation_shape shp, relation_dtype dt, relation_kernel kernel,
                                  int* dev_status, relation_stream_t stream) {
  relation_status st;
  if ((st = check_shape(shp, dt)) != RELATION_OK) return st;
  if ((st = check_scalars(lambda, tau_s)) != RELATION_OK) return st;
  if ((st = check_ptrs({q, k, v, o, logz})) != RELATION_OK) return st;
  if (self_flow && (st = check_ptrs({self_flow})) != RELATION_OK) return st;
  if (dev_status && (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return RELATION_ERR_ALIGNMENT;
  const int fam = pick_family(kernel, dt, shp.d_h, false);
  if (fam == 0) return RELATION_ERR_UNSUPPORTED;
  Problem p = make_problem(shp, dt, lambda, tau_s, dev_status);
  p.q = q; p.k = k; p.v = v; p.out = o; p.logz = logz; p.fself = self_flow;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return from_cuda(fam == 2 ? rel::tc::launch_fwd(p, s) : rel::simt::launch_fwd(p, s));
}

relation_status relation_fwd_ex(const void* q, const void* k, const void* v, void* o, float* logz,
                                float lambda, float tau_s, relation_shape shp, relation_dtype dt,
                                relation_kernel kernel, int* dev_status, relation_stream_t stream) {
  return relation_fwd_flow(q, k, v, o, logz, nullptr, lambda, tau_s, shp, dt, kernel, dev_status,
                           stream);
}

relation_status relation_fwd(const void* q, const void* k, const void* v, void* o, float* logz,
                             float lambda, float tau_s, relation_shape shp, relation_dtype dt,
                             int* dev_status, relation_stream_t stream) {
  return relation_fwd_ex(q, k, v, o, logz, lambda, tau_s, shp, dt, RELATION_KERNEL_AUTO,
                         dev_status, stream);
}

relation_status relation_fwd_state(const void* q, const void* k, const void* v, float* m,
                                   float* l, float* z, relation_shape shp_q,
                                   relation_shape shp_kv, int causal, relation_dtype dt,
                                   int* dev_status, relation_stream_t stream) {
  relation_status st;
  if ((st = check_shape(shp_q, dt)) != RELATION_OK) return st;
  if ((st = check_shape(shp_kv, dt)) != RELATION_OK) return st;
  if (causal != 0 && causal != 1) return RELATION_ERR_INVALID_ARG;
  if (shp_kv.B != shp_q.B || shp_kv.H != shp_q.H || shp_kv.d_h != shp_q.d_h)
    return RELATION_ERR_INVALID_ARG;
  if (causal && shp_kv.T != shp_q.T) return RELATION_ERR_INVALID_ARG;
  if (!rel::tc::supports(dt, shp_q.d_h)) return RELATION_ERR_UNSUPPORTED;  // bf16 tiles
  if ((long long)((shp_q.T + 127) / 128) * shp_q.B * shp_q.H > 0x7fffffffLL)
    return RELATION_ERR_UNSUPPORTED;
  if ((st = check_ptrs({q, k, v, m, l, z})) != RELATION_OK) return st;
  if (dev_status && (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return RELATION_ERR_ALIGNMENT;
  Problem p = make_problem(shp_q, dt, 0.0f, 1.0f, dev_status);
  p.q = q; p.k = k; p.v = v;
  rel::StateArgs sa{};
  sa.causal = causal;
  sa.Tk = shp_kv.T;
  sa.k_sB = shp_kv.sB; sa.k_sT = shp_kv.sT; sa.k_sH = shp_kv.sH;
  sa.m = m; sa.l = l; sa.z = z;
  return from_cuda(rel::tc::launch_fwd_state(p, sa, reinterpret_cast<cudaStream_t>(stream)));
}

relation_status relation_state_merge(float* m, float* l, float* z, const float* m2,
                                     const float* l2, const float* z2, relation_shape shp,
                                     relation_stream_t stream) {
  if (shp.B < 1 || shp.T < 1 || shp.H < 1) return RELATION_ERR_INVALID_ARG;
  if (shp.d_h < 4 || shp.d_h > 128 || shp.d_h % 4) return RELATION_ERR_UNSUPPORTED;
  relation_status st;
  if ((st = check_ptrs({m, l, z, m2, l2, z2})) != RELATION_OK) return st;
  const long long rows = (long long)shp.B * shp.H * shp.T;
  return from_cuda(rel::launch_state_merge(m, l, z, m2, l2, z2, rows, shp.d_h,
                                           reinterpret_cast<cudaStream_t>(stream)));
}

relation_status relation_state_finish(const void* q, const void* k, const void* v,
                                      const float* m, const float* l, const float* z, void* o,
                                      float* logz, float* self_flow, float lambda, float tau_s,
                                      long long pos0, relation_shape shp, relation_dtype dt,
                                      relation_stream_t stream) {
  relation_status st;
  if ((st = check_shape(shp, dt)) != RELATION_OK) return st;
  if ((st = check_scalars(lambda, tau_s)) != RELATION_OK) return st;
  if (pos0 < 0) return RELATION_ERR_INVALID_ARG;
  if (shp.d_h < 4 || shp.d_h > 128 || shp.d_h % 4) return RELATION_ERR_UNSUPPORTED;
  if ((st = check_ptrs({q, k, v, m, l, z, o, logz})) != RELATION_OK) return st;
  if (self_flow && (st = check_ptrs({self_flow})) != RELATION_OK) return st;
  Problem p = make_problem(shp, dt, lambda, tau_s, nullptr);
  p.q = q; p.k = k; p.v = v; p.out = o; p.logz = logz; p.fself = self_flow;
  return from_cuda(rel::launch_state_finish(p, m, l, z, pos0,
                                            reinterpret_cast<cudaStream_t>(stream)));
}

relation_status relation_linear_fwd(const void* p1, const void* p2, const void* v,
                                   const float* alpha, void* y, float tau_s, relation_shape shp,
                                   relation_dtype dt, int* dev_status, relation_stream_t stream) {
  return relation_linear_fwd_ex(p1, p2, v, alpha, y, tau_s, shp, dt, RELATION_KERNEL_AUTO,
                                dev_status, stream);
}

relation_status relation_linear_fwd_ex(const void* p1, const void* p2, const void* v,
                                      const float* alpha, void* y, float tau_s,
                                      relation_shape shp, relation_dtype dt,
                                      relation_kernel kernel, int* dev_status,
                                      relation_stream_t stream) {
  relation_status st;
  if (kernel != RELATION_KERNEL_AUTO && kernel != RELATION_KERNEL_SIMT &&
      kernel != RELATION_KERNEL_TCGEN05)
    return RELATION_ERR_INVALID_ARG;
  if (dt != RELATION_F32 && dt != RELATION_BF16) return RELATION_ERR_INVALID_ARG;
  if (shp.B < 1 || shp.T < 1 || shp.H < 1 || shp.d_h < 1) return RELATION_ERR_INVALID_ARG;
  if (shp.sB < 1 || shp.sT < 1 || shp.sH < 1) return RELATION_ERR_INVALID_ARG;
  if (!rel::linear_supports(dt, shp.d_h)) return RELATION_ERR_UNSUPPORTED;
  // grid: up to 8 column splits per head
  if ((long long)shp.B * shp.H * 8 > 0x7fffffffLL) return RELATION_ERR_UNSUPPORTED;
  // 4-element vector loads of every token row (alpha is fp32 with the same strides)
  if (shp.sB % 4 || shp.sT % 4 || shp.sH % 4) return RELATION_ERR_ALIGNMENT;
  if (!isfinite(tau_s) || !(tau_s > 0.0f)) return RELATION_ERR_INVALID_ARG;
  if ((st = check_ptrs({p1, p2, v, alpha, y})) != RELATION_OK) return st;
  if (dev_status && (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return RELATION_ERR_ALIGNMENT;
  rel::LinearProblem p{};
  p.p1 = p1; p.p2 = p2; p.v = v; p.alpha = alpha; p.y = y; p.dev_status = dev_status;
  p.tau_s = tau_s; p.B = shp.B; p.T = shp.T; p.H = shp.H; p.d = shp.d_h;
  p.sB = shp.sB; p.sT = shp.sT; p.sH = shp.sH; p.dtype = dt;
  const bool tc = rel::linear_tc_supports(p);
  if (kernel == RELATION_KERNEL_TCGEN05 && !tc)
    return (dt == RELATION_BF16 && (shp.d_h == 64 || shp.d_h == 128)) ? RELATION_ERR_ALIGNMENT
                                                                     : RELATION_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (tc && kernel != RELATION_KERNEL_SIMT)
    return from_cuda(rel::launch_linear_tc_fwd(p, nullptr, s));
  return from_cuda(rel::launch_linear_fwd(p, s));
}

size_t relation_linear_fwd_workspace_size(relation_shape shp, relation_dtype dt) {
  if (dt != RELATION_BF16 || shp.B < 1 || shp.T < 1 || shp.H < 1) return 0;
  rel::LinearProblem p{};
  p.B = shp.B; p.T = shp.T; p.H = shp.H; p.d = shp.d_h;
  p.sB = shp.sB; p.sT = shp.sT; p.sH = shp.sH; p.dtype = dt;
  return rel::linear_tc_workspace_bytes(p);
}

relation_status relation_linear_fwd_ws(const void* p1, const void* p2, const void* v,
                                      const float* alpha, void* y, float tau_s,
                                      relation_shape shp, relation_dtype dt, void* workspace,
                                      size_t ws_bytes, int* dev_status,
                                      relation_stream_t stream) {
  const size_t need = relation_linear_fwd_workspace_size(shp, dt);
  if (need == 0)  // no chunked kernel for this request: the regular entry point decides
    return relation_linear_fwd_ex(p1, p2, v, alpha, y, tau_s, shp, dt, RELATION_KERNEL_AUTO,
                                  dev_status, stream);
  if (!workspace || ws_bytes < need) return RELATION_ERR_WORKSPACE;
  if (!aligned16(workspace)) return RELATION_ERR_ALIGNMENT;
  int dev = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return RELATION_ERR_CUDA;
  const long long ctas = (long long)shp.B * shp.H * (shp.d_h / 64);
  // enough (head, column) pairs for the sequential walk (measured on GB300: 96 pairs on 152
  // SMs still favour it, 0.14 against 0.19 ms; 12 pairs at T = 32768 take 1.9 ms against 0.38)
  if (2 * ctas >= nsm)
    return relation_linear_fwd_ex(p1, p2, v, alpha, y, tau_s, shp, dt, RELATION_KERNEL_TCGEN05,
                                  dev_status, stream);
  relation_status st;
  if ((st = check_ptrs({p1, p2, v, alpha, y})) != RELATION_OK) return st;
  if (!isfinite(tau_s) || !(tau_s > 0.0f)) return RELATION_ERR_INVALID_ARG;
  if (dev_status && (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return RELATION_ERR_ALIGNMENT;
  if ((long long)ctas * ((shp.T + 127) / 128) > 0x7fffffffLL) return RELATION_ERR_UNSUPPORTED;
  rel::LinearProblem p{};
  p.p1 = p1; p.p2 = p2; p.v = v; p.alpha = alpha; p.y = y; p.dev_status = dev_status;
  p.tau_s = tau_s; p.B = shp.B; p.T = shp.T; p.H = shp.H; p.d = shp.d_h;
  p.sB = shp.sB; p.sT = shp.sT; p.sH = shp.sH; p.dtype = dt;
  return from_cuda(rel::launch_linear_tc_fwd(p, workspace, reinterpret_cast<cudaStream_t>(stream)));
}

namespace {

// The kernel family a backward request runs on (SIMT or TCGEN05), or -1 when the request
// is not served: the arguments' shapes and dtypes only, no pointers.
int linear_bwd_family(const relation_shape& shp, relation_dtype dt, relation_kernel kernel,
                      relation_status* why) {
  *why = RELATION_OK;
  if (kernel != RELATION_KERNEL_AUTO && kernel != RELATION_KERNEL_SIMT &&
      kernel != RELATION_KERNEL_TCGEN05) { *why = RELATION_ERR_INVALID_ARG; return -1; }
  if (dt != RELATION_F32 && dt != RELATION_BF16) { *why = RELATION_ERR_INVALID_ARG; return -1; }
  if (shp.B < 1 || shp.T < 1 || shp.H < 1 || shp.d_h < 1) { *why = RELATION_ERR_INVALID_ARG; return -1; }
  if (shp.sB < 1 || shp.sT < 1 || shp.sH < 1) { *why = RELATION_ERR_INVALID_ARG; return -1; }
  if (!rel::linear_supports(dt, shp.d_h)) { *why = RELATION_ERR_UNSUPPORTED; return -1; }
  // grid: up to 8 column splits per head
  if ((long long)shp.B * shp.H * 8 > 0x7fffffffLL) { *why = RELATION_ERR_UNSUPPORTED; return -1; }
  // 4-element vector loads of every token row (alpha is fp32 with the same strides)
  if (shp.sB % 4 || shp.sT % 4 || shp.sH % 4) { *why = RELATION_ERR_ALIGNMENT; return -1; }
  rel::LinearProblem p{};
  p.B = shp.B; p.T = shp.T; p.H = shp.H; p.d = shp.d_h;
  p.sB = shp.sB; p.sT = shp.sT; p.sH = shp.sH; p.dtype = dt;
  const bool tc = rel::linear_tc_bwd_supports(p) &&
                  (long long)shp.B * shp.H * ((shp.T + 127) / 128) <= 0x7fffffffLL;
  if (kernel == RELATION_KERNEL_TCGEN05 && !tc) {
    *why = (dt == RELATION_BF16 && shp.d_h == 64 && (shp.sB % 8 || shp.sT % 8 || shp.sH % 8))
               ? RELATION_ERR_ALIGNMENT : RELATION_ERR_UNSUPPORTED;
    return -1;
  }
  return (tc && kernel != RELATION_KERNEL_SIMT) ? (int)RELATION_KERNEL_TCGEN05
                                                : (int)RELATION_KERNEL_SIMT;
}

size_t linear_bwd_bytes(const relation_shape& shp, relation_dtype dt, int family) {
  if (family == (int)RELATION_KERNEL_SIMT)
    return rel::linear_bwd_workspace_bytes(shp.B, shp.H, shp.T, shp.d_h);
  rel::LinearProblem p{};
  p.B = shp.B; p.T = shp.T; p.H = shp.H; p.d = shp.d_h;
  p.sB = shp.sB; p.sT = shp.sT; p.sH = shp.sH; p.dtype = dt;
  return rel::linear_tc_bwd_workspace_bytes(p);
}

}  // namespace

size_t relation_linear_bwd_ex_workspace_size(relation_shape shp, relation_dtype dt,
                                             relation_kernel kernel) {
  relation_status why;
  const int fam = linear_bwd_family(shp, dt, kernel, &why);
  return fam < 0 ? 0 : linear_bwd_bytes(shp, dt, fam);
}

size_t relation_linear_bwd_workspace_size(relation_shape shp, relation_dtype dt) {
  return relation_linear_bwd_ex_workspace_size(shp, dt, RELATION_KERNEL_AUTO);
}

relation_status relation_linear_bwd(const void* p1, const void* p2, const void* v,
                                   const float* alpha, const void* dy, void* dp1, void* dp2,
                                   void* dv, float* dalpha, float tau_s, relation_shape shp,
                                   relation_dtype dt, void* workspace, size_t ws_bytes,
                                   int* dev_status, relation_stream_t stream) {
  return relation_linear_bwd_ex(p1, p2, v, alpha, dy, dp1, dp2, dv, dalpha, tau_s, shp, dt,
                                RELATION_KERNEL_AUTO, workspace, ws_bytes, dev_status, stream);
}

relation_status relation_linear_bwd_ex(const void* p1, const void* p2, const void* v,
                                      const float* alpha, const void* dy, void* dp1, void* dp2,
                                      void* dv, float* dalpha, float tau_s, relation_shape shp,
                                      relation_dtype dt, relation_kernel kernel, void* workspace,
                                      size_t ws_bytes, int* dev_status,
                                      relation_stream_t stream) {
  relation_status st;
  const int fam = linear_bwd_family(shp, dt, kernel, &st);
  if (fam < 0) return st;
  if (!isfinite(tau_s) || !(tau_s > 0.0f)) return RELATION_ERR_INVALID_ARG;
  if ((st = check_ptrs({p1, p2, v, alpha, dy, dp1, dp2, dv, dalpha, workspace})) != RELATION_OK)
    return st;
  if (dev_status && (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return RELATION_ERR_ALIGNMENT;
  if (ws_bytes < linear_bwd_bytes(shp, dt, fam)) return RELATION_ERR_WORKSPACE;
  if (!aligned16(workspace)) return RELATION_ERR_ALIGNMENT;
  rel::LinearProblem p{};
  p.p1 = p1; p.p2 = p2; p.v = v; p.alpha = alpha; p.dy = dy;
  p.dp1 = dp1; p.dp2 = dp2; p.dv = dv; p.dalpha = dalpha; p.workspace = workspace;
  p.dev_status = dev_status; p.tau_s = tau_s;
  p.B = shp.B; p.T = shp.T; p.H = shp.H; p.d = shp.d_h;
  p.sB = shp.sB; p.sT = shp.sT; p.sH = shp.sH; p.dtype = dt;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (fam == (int)RELATION_KERNEL_TCGEN05) return from_cuda(rel::launch_linear_tc_bwd(p, s));
  return from_cuda(rel::launch_linear_bwd(p, s));
}

namespace {

relation_status check_layer(const relation_shape& shp, relation_dtype dt, int pairing,
                            float rope_base) {
  if (dt != RELATION_F32 && dt != RELATION_BF16) return RELATION_ERR_INVALID_ARG;
  if (shp.B < 1 || shp.T < 1 || shp.H < 1 || shp.d_h < 1) return RELATION_ERR_INVALID_ARG;
  if (shp.sB < 1 || shp.sT < 1 || shp.sH < 1) return RELATION_ERR_INVALID_ARG;
  if (pairing != 0 && pairing != 1) return RELATION_ERR_INVALID_ARG;
  if (!isfinite(rope_base) || !(rope_base > 0.0f)) return RELATION_ERR_INVALID_ARG;
  if (!rel::layer_supports(dt, shp.d_h, shp.H)) return RELATION_ERR_UNSUPPORTED;
  if ((long long)shp.B * ((shp.T + 15) / 16) > 0x7fffffffLL) return RELATION_ERR_UNSUPPORTED;
  const long long vec = 16 / (long long)elem_size(dt);
  if (shp.sB % vec || shp.sT % vec || shp.sH % vec) return RELATION_ERR_ALIGNMENT;
  return RELATION_OK;
}

rel::LayerProblem layer_problem(const relation_shape& shp, relation_dtype dt, int pairing,
                                float rope_base, const float* theta) {
  rel::LayerProblem p{};
  p.theta = theta; p.pairing = pairing; p.rope_base = rope_base;
  p.B = shp.B; p.T = shp.T; p.H = shp.H; p.d = shp.d_h;
  p.sB = shp.sB; p.sT = shp.sT; p.sH = shp.sH; p.dtype = dt;
  return p;
}

}  // namespace

relation_status relation_layer_prep(const void* p1, const void* p2, const void* info,
                                    const float* theta, int pairing, float rope_base, void* q,
                                    void* k, void* v, relation_shape shp, relation_dtype dt,
                                    relation_stream_t stream) {
  relation_status st;
  if ((st = check_layer(shp, dt, pairing, rope_base)) != RELATION_OK) return st;
  if ((st = check_ptrs({p1, p2, info, q, k, v})) != RELATION_OK) return st;
  if (!theta || (reinterpret_cast<uintptr_t>(theta) & 3u)) return RELATION_ERR_INVALID_ARG;
  rel::LayerProblem p = layer_problem(shp, dt, pairing, rope_base, theta);
  p.in1 = p1; p.in2 = p2; p.in3 = info; p.out1 = q; p.out2 = k; p.out3 = v;
  return from_cuda(rel::launch_layer_prep(p, reinterpret_cast<cudaStream_t>(stream)));
}

size_t relation_layer_grad_workspace_size(relation_shape shp, relation_dtype dt) {
  if (check_layer(shp, dt, 0, 1.0f) != RELATION_OK) return 0;
  return rel::layer_grad_workspace_bytes(shp.B, shp.T, shp.H);
}

relation_status relation_layer_grad(const void* dq, const void* dk, const void* dv,
                                    const void* info, const float* theta, int pairing,
                                    float rope_base, void* dp1, void* dp2, void* dinfo,
                                    float* dtheta, relation_shape shp, relation_dtype dt,
                                    void* workspace, size_t ws_bytes, relation_stream_t stream) {
  relation_status st;
  if ((st = check_layer(shp, dt, pairing, rope_base)) != RELATION_OK) return st;
  if ((st = check_ptrs({dq, dk, dv, info, dp1, dp2, dinfo, workspace})) != RELATION_OK) return st;
  if (!theta || (reinterpret_cast<uintptr_t>(theta) & 3u)) return RELATION_ERR_INVALID_ARG;
  if (!dtheta || (reinterpret_cast<uintptr_t>(dtheta) & 3u)) return RELATION_ERR_INVALID_ARG;
  if (ws_bytes < rel::layer_grad_workspace_bytes(shp.B, shp.T, shp.H)) return RELATION_ERR_WORKSPACE;
  rel::LayerProblem p = layer_problem(shp, dt, pairing, rope_base, theta);
  p.in1 = dq; p.in2 = dk; p.in3 = dv; p.in4 = info;
  p.out1 = dp1; p.out2 = dp2; p.out3 = dinfo;
  p.dtheta = dtheta; p.dtheta_part = reinterpret_cast<float*>(workspace);
  return from_cuda(rel::launch_layer_grad(p, reinterpret_cast<cudaStream_t>(stream)));
}

size_t relation_decode_workspace_size(relation_shape cache, relation_dtype dt) {
  if (dt != RELATION_F32 && dt != RELATION_BF16) return 0;
  if (cache.B < 1 || cache.T < 1 || cache.H < 1 || cache.d_h < 1 || cache.d_h > 128) return 0;
  return rel::decode_workspace_bytes(cache.B, cache.H, cache.T);
}

relation_status relation_decode(const void* q, const void* k_cache, const void* v_cache,
                                const int* lengths, void* o, float* logz, float lambda,
                                float tau_s, relation_shape cache, long long q_sB, long long q_sH,
                                relation_dtype dt, void* workspace, size_t ws_bytes,
                                int* dev_status, relation_stream_t stream) {
  relation_status st;
  if (dt != RELATION_F32 && dt != RELATION_BF16) return RELATION_ERR_INVALID_ARG;
  if (cache.B < 1 || cache.T < 1 || cache.H < 1 || cache.d_h < 1) return RELATION_ERR_INVALID_ARG;
  if (cache.d_h > 128) return RELATION_ERR_UNSUPPORTED;
  if ((long long)cache.B * cache.H > 0x7fffffffLL) return RELATION_ERR_UNSUPPORTED;
  if (cache.sB < 1 || cache.sT < 1 || cache.sH < 1 || q_sB < 1 || q_sH < 1)
    return RELATION_ERR_INVALID_ARG;
  if ((st = check_scalars(lambda, tau_s)) != RELATION_OK) return st;
  if ((st = check_ptrs({q, k_cache, v_cache, lengths, o, logz, workspace})) != RELATION_OK)
    return st;
  if (dev_status && (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return RELATION_ERR_ALIGNMENT;
  if (ws_bytes < rel::decode_workspace_bytes(cache.B, cache.H, cache.T))
    return RELATION_ERR_WORKSPACE;
  rel::DecodeProblem p{};
  p.q = q; p.k = k_cache; p.v = v_cache; p.lengths = lengths; p.out = o; p.logz = logz;
  p.dev_status = dev_status;
  p.lambda = lambda; p.tau_s = tau_s; p.inv_sqrt_d = 1.0f / sqrtf((float)cache.d_h);
  p.B = cache.B; p.T = cache.T; p.H = cache.H; p.d = cache.d_h;
  p.sB = cache.sB; p.sT = cache.sT; p.sH = cache.sH; p.qsB = q_sB; p.qsH = q_sH;
  p.dtype = dt;
  if (rel::decode_chunks(cache.T) > 65535) return RELATION_ERR_UNSUPPORTED;  // grid.y limit
  return from_cuda(rel::launch_decode(p, workspace, reinterpret_cast<cudaStream_t>(stream)));
}

size_t relation_bwd_workspace_size(relation_shape shp, relation_dtype dt) {
  if (check_shape(shp, dt) != RELATION_OK) return 0;
  return rel::bwd_workspace_bytes(shp.B, shp.H, shp.T, shp.d_h);
}

relation_status relation_bwd_stages(const void* q, const void* k, const void* v, const void* o,
                                    const void* dout, const float* logz, void* dq, void* dk,
                                    void* dv, float* dlambda, float lambda, float tau_s,
                                    relation_shape shp, relation_dtype dt, void* workspace,
                                    size_t ws_bytes, relation_kernel kernel, unsigned stages,
                                    int* dev_status, relation_stream_t stream) {
  relation_status st;
  if (stages == 0 || (stages & ~7u)) return RELATION_ERR_INVALID_ARG;
  if ((st = check_shape(shp, dt)) != RELATION_OK) return st;
  if ((st = check_scalars(lambda, tau_s)) != RELATION_OK) return st;
  if ((st = check_ptrs({q, k, v, o, dout, logz, dq, dk, dv})) != RELATION_OK) return st;
  if (!dlambda) return RELATION_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(dlambda) & 3u) return RELATION_ERR_ALIGNMENT;
  if (dev_status && (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return RELATION_ERR_ALIGNMENT;
  const size_t need = rel::bwd_workspace_bytes(shp.B, shp.H, shp.T, shp.d_h);
  if (!workspace || ws_bytes < need) return RELATION_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(workspace) & 255u) return RELATION_ERR_ALIGNMENT;
  const int fam = pick_family(kernel, dt, shp.d_h, true);
  if (fam == 0) return RELATION_ERR_UNSUPPORTED;

  Problem p = make_problem(shp, dt, lambda, tau_s, dev_status);
  p.q = q; p.k = k; p.v = v; p.o = o; p.dout = dout; p.logz_in = logz;
  p.dq = dq; p.dk = dk; p.dv = dv; p.dlambda = dlambda;
  rel::BwdWorkspace ws = rel::carve_workspace(workspace, shp.B, shp.H, shp.T, shp.d_h);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (fam == 2) return from_cuda(rel::tc::launch_bwd(p, ws, stages, s));
  cudaError_t e = cudaSuccess;
  if ((stages & 1) && (e = rel::bwd_common::launch_pre(p, ws, s)) != cudaSuccess) return from_cuda(e);
  if ((stages & 2) && (e = rel::simt::launch_bwd(p, ws, s)) != cudaSuccess) return from_cuda(e);
  if (stages & 4) e = rel::bwd_common::launch_dlambda(p, ws, rel::simt::main_ctas(p), s);
  return from_cuda(e);
}

relation_status relation_bwd_ex(const void* q, const void* k, const void* v, const void* o,
                                const void* dout, const float* logz, void* dq, void* dk, void* dv,
                                float* dlambda, float lambda, float tau_s, relation_shape shp,
                                relation_dtype dt, void* workspace, size_t ws_bytes,
                                relation_kernel kernel, int* dev_status, relation_stream_t stream) {
  return relation_bwd_stages(q, k, v, o, dout, logz, dq, dk, dv, dlambda, lambda, tau_s, shp, dt,
                             workspace, ws_bytes, kernel, RELATION_BWD_ALL, dev_status, stream);
}

relation_status relation_bwd(const void* q, const void* k, const void* v, const void* o,
                             const void* dout, const float* logz, void* dq, void* dk, void* dv,
                             float* dlambda, float lambda, float tau_s, relation_shape shp,
                             relation_dtype dt, void* workspace, size_t ws_bytes,
                             int* dev_status, relation_stream_t stream) {
  return relation_bwd_ex(q, k, v, o, dout, logz, dq, dk, dv, dlambda, lambda, tau_s, shp, dt,
                         workspace, ws_bytes, RELATION_KERNEL_AUTO, dev_status, stream);
}

const char* relation_status_string(relation_status s) {
  switch (s) {
    case RELATION_OK: return "RELATION_OK";
    case RELATION_ERR_INVALID_ARG: return "RELATION_ERR_INVALID_ARG";
    case RELATION_ERR_UNSUPPORTED: return "RELATION_ERR_UNSUPPORTED";
    case RELATION_ERR_ALIGNMENT: return "RELATION_ERR_ALIGNMENT";
    case RELATION_ERR_WORKSPACE: return "RELATION_ERR_WORKSPACE";
    case RELATION_ERR_CUDA: return "RELATION_ERR_CUDA";
    case RELATION_ERR_TIMEOUT: return "RELATION_ERR_TIMEOUT";
  }
  return "RELATION_ERR_UNKNOWN";
}

const char* relation_last_cuda_error(void) {
  snprintf(g_last_message, sizeof(g_last_message), "%s%s%s", g_last_where,
           g_last_where[0] ? ": " : "", cudaGetErrorString(g_last_cuda_error));
  return g_last_message;
}

int relation_version(void) { return (1 << 16) | 0; }

int relation_launch_count(relation_dtype dt, int d_h, relation_kernel kernel, int backward) {
  if (dt != RELATION_F32 && dt != RELATION_BF16) return 0;
  const int fam = pick_family(kernel, dt, d_h, backward != 0);
  if (fam == 0) return 0;
  if (!backward) return 1;
  // SIMT: row pre-pass, dK/dV kernel, dQ kernel, dlambda reduction;
  // tcgen05: row pass, tile kernel, finalisation (dQ conversion + dlambda reduction)
  return fam == 2 ? rel::tc::bwd_launches() : 4;
}

relation_status relation_selftest_wait_timeout(int* dev_status, int timeout_us,
                                               relation_stream_t stream) {
  if (!dev_status || timeout_us < 1 || timeout_us > 100000) return RELATION_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(dev_status) & 3u) return RELATION_ERR_ALIGNMENT;
  return from_cuda(
      rel::launch_selftest_wait(dev_status, timeout_us, reinterpret_cast<cudaStream_t>(stream)));
}

}  // extern "C"
