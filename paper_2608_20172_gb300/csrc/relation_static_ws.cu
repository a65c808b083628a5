// relation_static_ws.cu -- relation_bwd_static: the backward without a caller workspace.
//
// Some callers cannot allocate device memory: code embedded in a runtime that owns the
// whole device memory budget through its own allocator (and forbids direct cudaMalloc),
// or code on a path where an allocation could fail or synchronise the device at a bad
// time.  This entry point runs the same backward as relation_bwd_ex, with its scratch
// taken from a fixed array that lives in this file for the lifetime of the process:
// RELATION_STATIC_SCRATCH_BYTES on every GPU that loads the library.
//
// Set-up: the first call on a device looks up that device's address of the array
// (cudaGetSymbolAddress, with the device current) and caches it; make that first call
// before any stream capture.  Nothing here allocates memory.
//
// The array is shared by every call and keeps the previous call's contents.  The
// backward's first stage (its row pass) writes every scratch element the later stages
// read, so nothing has to be cleared between calls.  Calls whose executions overlap on
// the GPU (different streams, or different host threads) race on the array: serialise
// them.
#include <mutex>

#include "kernels.h"
#include "relation.h"

namespace {

static __device__ __align__(256) unsigned char g_bwd_scratch[RELATION_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 256;
std::mutex g_setup_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Address of this device's copy of the array, looked up once per device.
cudaError_t scratch_address(void** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (!g_scratch_ptr[dev]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_bwd_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = ptr;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" relation_status relation_bwd_static(
    const void* q, const void* k, const void* v, const void* o, const void* dout,
    const float* logz, void* dq, void* dk, void* dv, float* dlambda, float lambda, float tau_s,
    relation_shape shp, relation_dtype dt, relation_kernel kernel, int* dev_status,
    relation_stream_t stream) {
  const size_t need = relation_bwd_workspace_size(shp, dt);
  if (need == 0)  // invalid shape or dtype: let the regular entry point report which
    return relation_bwd_ex(q, k, v, o, dout, logz, dq, dk, dv, dlambda, lambda, tau_s, shp, dt,
                           nullptr, 0, kernel, dev_status, stream);
  if (need > (size_t)RELATION_STATIC_SCRATCH_BYTES) return RELATION_ERR_WORKSPACE;
  void* ws = nullptr;
  if (scratch_address(&ws) != cudaSuccess) return RELATION_ERR_CUDA;
  return relation_bwd_ex(q, k, v, o, dout, logz, dq, dk, dv, dlambda, lambda, tau_s, shp, dt, ws,
                         (size_t)RELATION_STATIC_SCRATCH_BYTES, kernel, dev_status, stream);
}
