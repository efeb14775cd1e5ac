// k_attn.cu -- scattered-query causal GQA attention over the paged cache.
// Row i (position pos[i]) attends keys 0..pos[i] of its document's cache at
// `layer`; keys of repaired rows were written before this launch (so every
// row of the pass sees the fresh K/V of the others), all others are stale.
#include <math.h>

#include "kvr_internal.cuh"

namespace kvr {
namespace {

template <typename T>
__device__ __forceinline__ float ldv(const T *p, size_t i);
template <>
__device__ __forceinline__ float ldv<float>(const float *p, size_t i) { return p[i]; }
template <>
__device__ __forceinline__ float ldv<__nv_bfloat16>(const __nv_bfloat16 *p, size_t i) {
  return __bfloat162float(p[i]);
}

// One warp per (row, query head); lanes split head_dim (VPL values each);
// online softmax over the keys in position order.
template <typename T, int VPL>
__global__ void __launch_bounds__(128)
    k_attn_simt(const float *q, const int32_t *pos, int M, int H, int G, int layer,
                const KVView *views, const int32_t *rowdoc, KVView single, T *out, float scale) {
  int w = blockIdx.x * 4 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (w >= M * H) return;
  const int dh = 32 * VPL;
  int i = w / H, hh = w % H, g = hh / (H / G);
  int p = pos[i];
  KVView v = views ? views[rowdoc[i]] : single;
  const T *c = (const T *)v.pages;
  float qv[VPL], o[VPL];
#pragma unroll
  for (int e = 0; e < VPL; ++e) {
    qv[e] = q[(size_t)i * H * dh + (size_t)hh * dh + lane * VPL + e] * scale;
    o[e] = 0.f;
  }
  float mx = -INFINITY, l = 0.f;
  for (int j = 0; j <= p; ++j) {
    size_t ko = v.offset(layer, 0, g, j) + lane * VPL;
    size_t vo = v.offset(layer, 1, g, j) + lane * VPL;
    float s = 0.f;
#pragma unroll
    for (int e = 0; e < VPL; ++e) s += qv[e] * ldv(c, ko + e);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    float mn = fmaxf(mx, s);
    float corr = expf(mx - mn);
    float pj = expf(s - mn);
    l = l * corr + pj;
#pragma unroll
    for (int e = 0; e < VPL; ++e) o[e] = o[e] * corr + pj * ldv(c, vo + e);
    mx = mn;
  }
  float inv = 1.0f / l;
#pragma unroll
  for (int e = 0; e < VPL; ++e) {
    size_t oi = (size_t)i * H * dh + (size_t)hh * dh + lane * VPL + e;
    if constexpr (sizeof(T) == 2)
      out[oi] = __float2bfloat16_rn(o[e] * inv);
    else
      out[oi] = o[e] * inv;
  }
}

template <typename T>
void attn_simt_dispatch(const float *q, const int32_t *pos, int M, const Dims &dm, int layer,
                        const KVView *views, const int32_t *rowdoc, KVView single, void *out,
                        cudaStream_t s) {
  int warps = M * dm.H;
  int blocks = (warps + 3) / 4;
  float scale = (float)(1.0 / sqrt((double)dm.dh));
  if (dm.dh == 64)
    k_attn_simt<T, 2><<<blocks, 128, 0, s>>>(q, pos, M, dm.H, dm.G, layer, views, rowdoc, single,
                                             (T *)out, scale);
  else
    k_attn_simt<T, 4><<<blocks, 128, 0, s>>>(q, pos, M, dm.H, dm.G, layer, views, rowdoc, single,
                                             (T *)out, scale);
}

}  // namespace

void launch_attention_simt(const float *q, const int32_t *pos, int M, const Dims &dm, int layer,
                           const KVView *views, const int32_t *rowdoc, KVView single, void *out,
                           cudaStream_t s) {
  if (M <= 0) return;
  if (dm.dtype == KVR_DTYPE_BF16)
    attn_simt_dispatch<__nv_bfloat16>(q, pos, M, dm, layer, views, rowdoc, single, out, s);
  else
    attn_simt_dispatch<float>(q, pos, M, dm, layer, views, rowdoc, single, out, s);
}

}  // namespace kvr
