// relation_static_ws.cu -- relation_bwd_static: the backward without a caller workspace.
//
// Some callers cannot allocate device memory: code embedded in a runtime that owns the
// whole device memory budget through its own allocator (and forbids direct cudaMalloc),
// or code on a path where an allocation could fail or synchronise the device at a bad
// time.  This entry point runs the same backward as relation_bwd_ex, with its scratch
// taken from a fixed array that lives in this file for the lifetime of the process:
// RELATION_STATIC_SCRATCH_BYTES on every GPU that loads the library.
//
// Device.  The operands must live on the device that is current on the calling thread:
// the array used is that device's copy, and a call whose q is on another device is
// rejected with RELATION_ERR_INVALID_ARG before anything is launched.
//
// Set-up.  Every call looks up the current device's address of the array
// (cudaGetSymbolAddress with that device current; cheap once the module is loaded, and
// never stale after a device reset).  Under CUDA's lazy module loading the first call on
// a device (or the library's first launch there) loads the module and commits the array's
// RELATION_STATIC_SCRATCH_BYTES at that moment, so a caller whose allocator already owns
// the memory budget should make a first call during set-up, before any stream capture;
// the same holds for the first call after a device reset.  No call allocates memory
// otherwise.
//
// The array is shared by every call and keeps the previous call's contents.  The
// backward's first stage (its row pass) writes every scratch element the later stages
// read, so nothing has to be cleared between calls.  Calls whose executions overlap on
// the GPU (different streams, or different host threads) race on the array: serialise
// them.
#include "kernels.h"
#include "relation.h"

namespace {

static __device__ __align__(256) unsigned char g_bwd_scratch[RELATION_STATIC_SCRATCH_BYTES];

// 1 when p is device (or managed) memory of device dev, else 0.
int on_device(const void* p, int dev) {
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    (void)cudaGetLastError();  // a pointer CUDA does not know: clear the (non-sticky) error
    return 0;
  }
  if (a.type != cudaMemoryTypeDevice && a.type != cudaMemoryTypeManaged) return 0;
  return a.device == dev ? 1 : 0;
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
  if (!q) return RELATION_ERR_INVALID_ARG;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return RELATION_ERR_CUDA;
  if (on_device(q, dev) != 1) return RELATION_ERR_INVALID_ARG;  // q is not on this device
  void* ws = nullptr;
  if (cudaGetSymbolAddress(&ws, g_bwd_scratch) != cudaSuccess) return RELATION_ERR_CUDA;
  return relation_bwd_ex(q, k, v, o, dout, logz, dq, dk, dv, dlambda, lambda, tau_s, shp, dt, ws,
                         (size_t)RELATION_STATIC_SCRATCH_BYTES, kernel, dev_status, stream);
}
