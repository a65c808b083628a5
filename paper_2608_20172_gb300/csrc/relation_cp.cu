// relation_cp.cu -- context parallelism of the forward: the merge of two Exchange summaries
// and the epilogue from a merged summary (App. A.3, the online update of (m, l, z) being
// associative; App. A.3.3-A.3.5 for the epilogue).
//
// A sequence split into shards of consecutive tokens: each shard's queries take the
// Exchange summary over their own earlier tokens (relation_tc_fwd.cu, MODE 1, causal) and
// over every earlier shard's keys (MODE 1, all keys), the summaries are merged, and the
// epilogue adds the Self entry and the count term with the shard's absolute positions.
//   merge:   M = max(m, m'),  l = e^{m - M} l + e^{m' - M} l',  z = e^{m - M} z + e^{m' - M} z'
//   finish:  S_i = sigmoid(q_i . k_i / (sqrt(d) tau_S)),  A_i = m + log l - lambda log i,
//            g = sigmoid(A - S),  Y_i = (1 - g) v_i + g z / l,  logZ_i = logaddexp(S, A),
//            and the empty history (l = 0): g = 0, Y_i = v_i, logZ_i = S_i.
// One warp per row (d_h <= 128: four columns per lane), memory-bound.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rel {
namespace cp {

// (m, l, z) <- merge with (m2, l2, z2); rows of d floats in z.  Every lane reads the row's
// scalars before lane 0 overwrites them.
__global__ void __launch_bounds__(256) merge_kernel(float* m, float* l, float* z, const float* m2,
                                                    const float* l2, const float* z2,
                                                    long long rows, int d) {
  const long long row = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const float ma = m[row], mb = m2[row], la = l[row], lb = l2[row];
  const float M = fmaxf(ma, mb);
  // an empty summary has m = -inf and l = 0, z = 0: its factor is 0
  const float fa = ma == -INFINITY ? 0.f : __expf(ma - M);
  const float fb = mb == -INFINITY ? 0.f : __expf(mb - M);
  const int c = lane * 4;
  if (c < d) {
    float4* za = reinterpret_cast<float4*>(z + row * d + c);
    const float4 x = *za, y = *reinterpret_cast<const float4*>(z2 + row * d + c);
    *za = make_float4(fa * x.x + fb * y.x, fa * x.y + fb * y.y, fa * x.z + fb * y.z,
                      fa * x.w + fb * y.w);
  }
  __syncwarp();
  if (lane == 0) {
    m[row] = M;
    l[row] = fa * la + fb * lb;
  }
}

template <typename T>
__device__ __forceinline__ float4 load4(const T* p);
template <>
__device__ __forceinline__ float4 load4<float>(const float* p) {
  return *reinterpret_cast<const float4*>(p);
}
template <>
__device__ __forceinline__ float4 load4<__nv_bfloat16>(const __nv_bfloat16* p) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
  const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
  return make_float4(a.x, a.y, b.x, b.y);
}
template <typename T>
__device__ __forceinline__ void store4(T* p, float4 v);
template <>
__device__ __forceinline__ void store4<float>(float* p, float4 v) {
  *reinterpret_cast<float4*>(p) = v;
}
template <>
__device__ __forceinline__ void store4<__nv_bfloat16>(__nv_bfloat16* p, float4 v) {
  *reinterpret_cast<uint2*>(p) = make_uint2(pack_bf16x2(v.x, v.y), pack_bf16x2(v.z, v.w));
}

// The epilogue of rows [0, T) of every head from their merged summary; the row's one-based
// position is pos0 + r + 1.
template <typename T>
__global__ void __launch_bounds__(256) finish_kernel(Problem p, const float* m, const float* l,
                                                     const float* z, long long pos0) {
  const long long row = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const long long rows = (long long)p.B * p.H * p.T;
  if (row >= rows) return;
  const int bh = (int)(row / p.T), r = (int)(row % p.T);
  const int b = bh / p.H, h = bh % p.H;
  const long long off = (long long)b * p.sB + (long long)h * p.sH + (long long)r * p.sT;
  const int c = lane * 4;
  const bool mine = c < p.d;
  float4 qv = make_float4(0.f, 0.f, 0.f, 0.f), kv = qv, vv = qv, zv = qv;
  if (mine) {
    qv = load4(static_cast<const T*>(p.q) + off + c);
    kv = load4(static_cast<const T*>(p.k) + off + c);
    vv = load4(static_cast<const T*>(p.v) + off + c);
    zv = *reinterpret_cast<const float4*>(z + row * p.d + c);
  }
  float u = qv.x * kv.x + qv.y * kv.y + qv.z * kv.z + qv.w * kv.w;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) u += __shfl_xor_sync(0xffffffffu, u, o);
  const float S = 1.0f / (1.0f + __expf(-(u * p.inv_sqrt_d) / p.tau_s));
  const float lr = l[row];
  float g = 0.f, inv_l = 0.f, lz = S, fself = 1.0f;
  if (lr > 0.f) {
    const float A = m[row] + __logf(lr) - p.lambda * __logf((float)(pos0 + r + 1));
    g = 1.0f / (1.0f + __expf(S - A));
    fself = 1.0f / (1.0f + __expf(A - S));
    const float hi = fmaxf(S, A), lo = fminf(S, A);
    lz = hi + log1pf(__expf(lo - hi));
    inv_l = 1.0f / lr;
  }
  if (mine)
    store4(static_cast<T*>(p.out) + off + c,
           make_float4(fmaf(g, zv.x * inv_l - vv.x, vv.x), fmaf(g, zv.y * inv_l - vv.y, vv.y),
                       fmaf(g, zv.z * inv_l - vv.z, vv.z), fmaf(g, zv.w * inv_l - vv.w, vv.w)));
  if (lane == 0) {
    p.logz[row] = lz;
    if (p.fself) p.fself[row] = fself;
  }
}

}  // namespace cp

cudaError_t launch_state_merge(float* m, float* l, float* z, const float* m2, const float* l2,
                               const float* z2, long long rows, int d, cudaStream_t s) {
  if (rows < 1 || d < 4 || d > 128 || d % 4) return cudaErrorInvalidValue;
  const long long blocks = (rows + 7) / 8;
  if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  cp::merge_kernel<<<(unsigned)blocks, 256, 0, s>>>(m, l, z, m2, l2, z2, rows, d);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) note_failure("state merge: launch");
  return e;
}

cudaError_t launch_state_finish(const Problem& p, const float* m, const float* l, const float* z,
                                long long pos0, cudaStream_t s) {
  const long long rows = (long long)p.B * p.H * p.T;
  if (rows < 1 || p.d < 4 || p.d > 128 || p.d % 4) return cudaErrorInvalidValue;
  const long long blocks = (rows + 7) / 8;
  if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  if (p.dtype == RELATION_BF16)
    cp::finish_kernel<__nv_bfloat16><<<(unsigned)blocks, 256, 0, s>>>(p, m, l, z, pos0);
  else
    cp::finish_kernel<float><<<(unsigned)blocks, 256, 0, s>>>(p, m, l, z, pos0);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) note_failure("state finish: launch");
  return e;
}

}  // namespace rel
