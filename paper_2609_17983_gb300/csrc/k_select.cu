// k_select.cu -- selector scores (Table 1) and the top-K rule.
//
// Scores become 64-bit keys, larger = better, indexed by j - s_end over the
// pool D = [s_end, n).  Key 0 marks a position the policy excludes
// (Structural: not a delimiter).  Top-K orders by key descending, then
// position ascending (ties to the lowest position), and returns the chosen
// positions ascending.
#include <math.h>

#include "kvr_internal.cuh"

namespace kvr {
namespace {

constexpr uint64_t GAMMA = 0x9E3779B97F4A7C15ull;

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Order-preserving map of a float to uint32 (NaN ranks as -inf).
__device__ __forceinline__ uint32_t ord_f32(float f) {
  if (isnan(f)) f = -INFINITY;
  uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// First delimiter position at or after s_end (n - 1 if none): the document
// boundary of EditLocal@boundary.  *bound must hold n - 1 on entry.
__global__ void k_first_delim(const int32_t *tokens, int n, int s_end, int delim, int *bound) {
  for (int j = s_end + blockIdx.x * blockDim.x + threadIdx.x; j < n; j += gridDim.x * blockDim.x)
    if (tokens[j] == delim) atomicMin(bound, j);
}

__global__ void k_scores_simple(int policy, const int32_t *tokens, int n, int s_end, int delim,
                                uint64_t seed, const int *bound, unsigned long long *keys) {
  int c = n - s_end;
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < c; t += gridDim.x * blockDim.x) {
    int j = s_end + t;
    unsigned long long k;
    if (policy == KVR_POLICY_RANDOM) {
      // first SplitMix64 output of state seed ^ (j * gamma)
      k = mix64((seed ^ ((uint64_t)j * GAMMA)) + GAMMA);
    } else {
      // nearest to the span first
      k = 0x100000000ull - (unsigned long long)t;
      if (policy == KVR_POLICY_STRUCTURAL && tokens[j] != delim) k = 0;
      if (policy == KVR_POLICY_EDITLOCAL_BOUNDARY && j > *bound) k = 0;
    }
    keys[t] = k;
  }
}

__global__ void k_float_keys(const float *scores, int n, int s_end, unsigned long long *keys) {
  int c = n - s_end;
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < c; t += gridDim.x * blockDim.x)
    keys[t] = (unsigned long long)ord_f32(scores[s_end + t]) + 1ull;
}

__device__ __forceinline__ bool better(unsigned long long ka, int ia, unsigned long long kb,
                                       int ib) {
  return ka > kb || (ka == kb && ia < ib);
}

// Single CTA bitonic sort of (key, index) pairs in shared memory.
__global__ void __launch_bounds__(1024)
    k_topk(const unsigned long long *keys, int c, int s_end, int K, int nonzero_only,
           int32_t *out, int32_t *count) {
  extern __shared__ unsigned char smem[];
  int P = 1;
  while (P < c) P <<= 1;
  unsigned long long *sk = (unsigned long long *)smem;
  int *si = (int *)(sk + P);
  __shared__ int n_elig;
  if (threadIdx.x == 0) n_elig = 0;
  __syncthreads();
  int local = 0;
  for (int t = threadIdx.x; t < P; t += blockDim.x) {
    if (t < c) {
      sk[t] = keys[t];
      si[t] = t;
      local += (!nonzero_only || keys[t] != 0ull) ? 1 : 0;
    } else {
      sk[t] = 0ull;
      si[t] = 0x7FFFFFFF;
    }
  }
  atomicAdd(&n_elig, local);
  __syncthreads();
  for (int k = 2; k <= P; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int t = threadIdx.x; t < P; t += blockDim.x) {
        int u = t ^ j;
        if (u > t) {
          bool up = (t & k) == 0;
          bool sw = up ? better(sk[u], si[u], sk[t], si[t]) : better(sk[t], si[t], sk[u], si[u]);
          if (sw) {
            unsigned long long tk = sk[t];
            sk[t] = sk[u];
            sk[u] = tk;
            int ti = si[t];
            si[t] = si[u];
            si[u] = ti;
          }
        }
      }
      __syncthreads();
    }
  }
  int cnt = min(K, n_elig);
  // chosen indices ascending: sort the first cnt indices (ascending) in place
  int Q = 1;
  while (Q < cnt) Q <<= 1;
  for (int t = threadIdx.x; t < Q; t += blockDim.x)
    if (t >= cnt) si[t] = 0x7FFFFFFF;
  __syncthreads();
  for (int k = 2; k <= Q; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int t = threadIdx.x; t < Q; t += blockDim.x) {
        int u = t ^ j;
        if (u > t) {
          bool up = (t & k) == 0;
          bool sw = up ? si[t] > si[u] : si[t] < si[u];
          if (sw) {
            int ti = si[t];
            si[t] = si[u];
            si[u] = ti;
          }
        }
      }
      __syncthreads();
    }
  }
  for (int t = threadIdx.x; t < cnt; t += blockDim.x) out[t] = s_end + si[t];
  if (threadIdx.x == 0) *count = cnt;
}

// Attention selector, one layer: block (span row r, query head hh) writes the
// softmax over the pool of q_{r,hh} . K_layer[j] / sqrt(dh) into
// probs[(r*H + hh) * c + (j - s_end)].
template <typename T>
__global__ void __launch_bounds__(256)
    k_attn_select_probs(const float *q, int H, int G, int dh, int layer, KVView v, int s_end,
                        int n, float *probs, float scale) {
  int r = blockIdx.x / H, hh = blockIdx.x % H, g = hh / (H / G);
  int c = n - s_end;
  extern __shared__ float qs[];
  __shared__ float red[32];
  for (int i = threadIdx.x; i < dh; i += blockDim.x)
    qs[i] = q[(size_t)r * H * dh + (size_t)hh * dh + i];
  __syncthreads();
  const T *kc = (const T *)v.pages;
  float *pr = probs + (size_t)blockIdx.x * c;
  float mx = -INFINITY;
  for (int t = threadIdx.x; t < c; t += blockDim.x) {
    size_t o = v.offset(layer, 0, g, s_end + t);
    float s = 0.f;
    for (int i = 0; i < dh; ++i) {
      float kv;
      if constexpr (sizeof(T) == 2)
        kv = __bfloat162float(kc[o + i]);
      else
        kv = kc[o + i];
      s += qs[i] * kv;
    }
    s *= scale;
    pr[t] = s;
    mx = fmaxf(mx, s);
  }
  for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  __syncthreads();
  if (threadIdx.x < 32) {
    float t = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : -INFINITY;
    for (int off = 16; off > 0; off >>= 1) t = fmaxf(t, __shfl_xor_sync(0xffffffffu, t, off));
    if (threadIdx.x == 0) red[0] = t;
  }
  __syncthreads();
  mx = red[0];
  __syncthreads();
  float z = 0.f;
  for (int t = threadIdx.x; t < c; t += blockDim.x) {
    float e = expf(pr[t] - mx);
    pr[t] = e;
    z += e;
  }
  for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(0xffffffffu, z, off);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = z;
  __syncthreads();
  if (threadIdx.x < 32) {
    float t = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
    for (int off = 16; off > 0; off >>= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
    if (threadIdx.x == 0) red[0] = t;
  }
  __syncthreads();
  float inv = 1.0f / red[0];
  for (int t = threadIdx.x; t < c; t += blockDim.x) pr[t] *= inv;
}

// score[j] += sum over (row, head) of probs, in a fixed order.
__global__ void k_attn_select_accum(const float *probs, int RH, int c, int s_end, float *score) {
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < c; t += gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int rh = 0; rh < RH; ++rh) s += probs[(size_t)rh * c + t];
    score[s_end + t] += s;
  }
}

// CacheBlend deviation: fresh layer-1 k (RoPE at the row's position) and v
// from qkv, rounded to the cache dtype, against the stale cache entries:
// score[pos] = ||dk||_2 + ||dv||_2 over all kv heads and dims.
template <typename T>
__global__ void __launch_bounds__(256)
    k_kv_deviation(const float *qkv, const float2 *rope, const int32_t *pos, int H, int G, int dh,
                   KVView v, float *score) {
  int i = blockIdx.x;
  int p = pos[i];
  int half = dh / 2, Nqkv = (H + 2 * G) * dh;
  const float *x = qkv + (size_t)i * Nqkv;
  const T *c = (const T *)v.pages;
  float dk = 0.f, dv = 0.f;
  for (int e = threadIdx.x; e < G * half; e += blockDim.x) {
    int g = e / half, t = e % half;
    float2 cs = rope[(size_t)p * half + t];
    float k1 = x[(H + g) * dh + t], k2 = x[(H + g) * dh + t + half];
    float r1 = k1 * cs.x - k2 * cs.y, r2 = k2 * cs.x + k1 * cs.y;
    float v1 = x[(H + G + g) * dh + t], v2 = x[(H + G + g) * dh + t + half];
    size_t ko = v.offset(1, 0, g, p), vo = v.offset(1, 1, g, p);
    float sk1, sk2, sv1, sv2;
    if constexpr (sizeof(T) == 2) {
      r1 = __bfloat162float(__float2bfloat16_rn(r1));
      r2 = __bfloat162float(__float2bfloat16_rn(r2));
      v1 = __bfloat162float(__float2bfloat16_rn(v1));
      v2 = __bfloat162float(__float2bfloat16_rn(v2));
      sk1 = __bfloat162float(c[ko + t]);
      sk2 = __bfloat162float(c[ko + t + half]);
      sv1 = __bfloat162float(c[vo + t]);
      sv2 = __bfloat162float(c[vo + t + half]);
    } else {
      sk1 = c[ko + t];
      sk2 = c[ko + t + half];
      sv1 = c[vo + t];
      sv2 = c[vo + t + half];
    }
    dk += (r1 - sk1) * (r1 - sk1) + (r2 - sk2) * (r2 - sk2);
    dv += (v1 - sv1) * (v1 - sv1) + (v2 - sv2) * (v2 - sv2);
  }
  __shared__ float rk[32], rv[32];
  for (int off = 16; off > 0; off >>= 1) {
    dk += __shfl_xor_sync(0xffffffffu, dk, off);
    dv += __shfl_xor_sync(0xffffffffu, dv, off);
  }
  if ((threadIdx.x & 31) == 0) {
    rk[threadIdx.x >> 5] = dk;
    rv[threadIdx.x >> 5] = dv;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float a = 0.f, b = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      a += rk[w];
      b += rv[w];
    }
    score[p] = sqrtf(a) + sqrtf(b);
  }
}

int grid_for(int n, int block) {
  int g = (n + block - 1) / block;
  return g < 1 ? 1 : (g > 4096 ? 4096 : g);
}

}  // namespace

void launch_scores_simple(int policy, const int32_t *tokens, int n, int s_end, int delim,
                          uint64_t seed, int *bound, unsigned long long *keys, cudaStream_t s) {
  int c = n - s_end;
  if (c <= 0) return;
  if (policy == KVR_POLICY_EDITLOCAL_BOUNDARY)
    k_first_delim<<<grid_for(c, 256), 256, 0, s>>>(tokens, n, s_end, delim, bound);
  k_scores_simple<<<grid_for(c, 256), 256, 0, s>>>(policy, tokens, n, s_end, delim, seed, bound,
                                                   keys);
}

void launch_float_keys(const float *scores, int n, int s_end, unsigned long long *keys,
                       cudaStream_t s) {
  int c = n - s_end;
  if (c <= 0) return;
  k_float_keys<<<grid_for(c, 256), 256, 0, s>>>(scores, n, s_end, keys);
}

// Top-K over c = n - s_end candidates (c <= 16384).  nonzero_only is
// encoded in the sign of K: K < 0 means "only nonzero keys are eligible".
// Returns nullptr on success, else what failed.
const char *launch_topk(const unsigned long long *keys, int n, int s_end, int K, int32_t *out,
                        int32_t *count, cudaStream_t s) {
  int c = n - s_end;
  int nonzero_only = K < 0 ? 1 : 0;
  if (K < 0) K = -K;
  if (c < 0) c = 0;
  int P = 1;
  while (P < c) P <<= 1;
  size_t smem = (size_t)P * (sizeof(unsigned long long) + sizeof(int));
  if (smem >= 32 * 1024) {  // the default 48 KB limit also covers static shared memory
    cudaError_t e = cudaFuncSetAttribute(k_topk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cudaGetErrorString(e);
  }
  k_topk<<<1, 1024, smem, s>>>(keys, c, s_end, K, nonzero_only, out, count);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

void launch_attn_select_scores(const float *q, int S, const Dims &dm, int layer, KVView v,
                               int s_end, int n, float *probs_ws, float *scores, cudaStream_t s) {
  int c = n - s_end;
  if (c <= 0 || S <= 0) return;
  float scale = (float)(1.0 / sqrt((double)dm.dh));
  size_t smem = (size_t)dm.dh * sizeof(float);
  if (dm.dtype == KVR_DTYPE_BF16)
    k_attn_select_probs<__nv_bfloat16><<<S * dm.H, 256, smem, s>>>(q, dm.H, dm.G, dm.dh, layer,
                                                                    v, s_end, n, probs_ws, scale);
  else
    k_attn_select_probs<float><<<S * dm.H, 256, smem, s>>>(q, dm.H, dm.G, dm.dh, layer, v, s_end,
                                                            n, probs_ws, scale);
  k_attn_select_accum<<<grid_for(c, 256), 256, 0, s>>>(probs_ws, S * dm.H, c, s_end, scores);
}

void launch_kv_deviation(const float *qkv, const float2 *rope, const int32_t *pos, int M,
                         const Dims &dm, KVView v, float *scores, cudaStream_t s) {
  if (M <= 0) return;
  if (dm.dtype == KVR_DTYPE_BF16)
    k_kv_deviation<__nv_bfloat16><<<M, 256, 0, s>>>(qkv, rope, pos, dm.H, dm.G, dm.dh, v, scores);
  else
    k_kv_deviation<float><<<M, 256, 0, s>>>(qkv, rope, pos, dm.H, dm.G, dm.dh, v, scores);
}

}  // namespace kvr
