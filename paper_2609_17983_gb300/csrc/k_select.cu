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

// Top-K of c (key, index) pairs, one CTA of TOPK_THREADS: key descending, ties to
// the lowest index, the chosen indices written ascending.  Instead of a sort,
// the K-th key T is found by an MSB-first radix select (8 bits per pass, a
// shared-memory histogram of the keys that still match the prefix); then
// every key above T is taken, and of the keys equal to T the lowest-indexed
// ones until K are taken.  Thread i owns the contiguous keys [i*E, (i+1)*E),
// so a block-wide scan of per-thread counts writes the output in index order.
constexpr int TOPK_THREADS = 1024;

__device__ __forceinline__ int block_excl_scan(int x, int *tmp) {
  // tmp: TOPK_THREADS / 32 ints
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int v = x;
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += y;
  }
  if (lane == 31) tmp[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int w = lane < TOPK_THREADS / 32 ? tmp[lane] : 0;
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < TOPK_THREADS / 32) tmp[lane] = w;
  }
  __syncthreads();
  const int before = (warp ? tmp[warp - 1] : 0) + v - x;
  __syncthreads();
  return before;
}

__global__ void __launch_bounds__(TOPK_THREADS)
    k_topk(const unsigned long long *keys, int c, int s_end, int K, int nonzero_only,
           int32_t *out, int32_t *count) {
  extern __shared__ unsigned long long sk[];  // c keys
  __shared__ int hist[256];
  __shared__ int scan_tmp[TOPK_THREADS / 32];
  __shared__ int s_elig, s_bin, s_above;
  const int tid = threadIdx.x;
  const int E = (c + TOPK_THREADS - 1) / TOPK_THREADS;
  const int t0 = min(c, tid * E), t1 = min(c, t0 + E);
  if (tid == 0) s_elig = 0;
  __syncthreads();
  int local = 0;
  for (int t = tid; t < c; t += TOPK_THREADS) {
    const unsigned long long k = keys[t];
    sk[t] = k;
    local += (!nonzero_only || k != 0ull) ? 1 : 0;
  }
  local += __shfl_xor_sync(0xffffffffu, local, 16);
  local += __shfl_xor_sync(0xffffffffu, local, 8);
  local += __shfl_xor_sync(0xffffffffu, local, 4);
  local += __shfl_xor_sync(0xffffffffu, local, 2);
  local += __shfl_xor_sync(0xffffffffu, local, 1);
  if ((tid & 31) == 0) atomicAdd(&s_elig, local);
  __syncthreads();
  const int cnt = min(K, s_elig);
  // radix select: prefix/mask of T, need = how many keys equal to the prefix
  // (so far) are still to be taken
  unsigned long long pref = 0ull, mask = 0ull;
  int need = cnt;
  for (int d = 56; d >= 0 && need > 0; d -= 8) {
    for (int i = tid; i < 256; i += TOPK_THREADS) hist[i] = 0;
    __syncthreads();
    for (int t = t0; t < t1; ++t) {
      const unsigned long long k = sk[t];
      if ((k & mask) == pref) atomicAdd(&hist[(int)(k >> d) & 255], 1);
    }
    __syncthreads();
    if (tid < 32) {
      // suffix sums over bins 255..0, 8 bins per lane (lane 0 holds 255..248)
      int loc[8], sum = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        loc[j] = hist[255 - (tid * 8 + j)];
        sum += loc[j];
      }
      int incl = sum;
      for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (tid >= o) incl += y;
      }
      int acc = incl - sum;  // keys in bins above this lane's first bin
      int found = -1, above = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (found < 0 && acc + loc[j] >= need) {
          found = 255 - (tid * 8 + j);
          above = acc;
        }
        acc += loc[j];
      }
      const unsigned ball = __ballot_sync(0xffffffffu, found >= 0);
      const int src = __ffs(ball) - 1;  // first lane (highest bins) that found it
      const int bin = __shfl_sync(0xffffffffu, found, src);
      const int ab = __shfl_sync(0xffffffffu, above, src);
      if (tid == 0) {
        s_bin = bin;
        s_above = ab;
      }
    }
    __syncthreads();
    pref |= (unsigned long long)s_bin << d;
    mask |= 0xFFull << d;
    need -= s_above;
    __syncthreads();
  }
  // T = pref (when cnt > 0): take keys > T, and the first `need` keys == T
  int gt = 0, eq = 0;
  if (cnt > 0)
    for (int t = t0; t < t1; ++t) {
      const unsigned long long k = sk[t];
      gt += k > pref ? 1 : 0;
      eq += k == pref ? 1 : 0;
    }
  const int eq_before = block_excl_scan(eq, scan_tmp);
  int take_eq = cnt > 0 ? min(eq, max(0, need - eq_before)) : 0;
  const int sel = gt + take_eq;
  int pos = block_excl_scan(sel, scan_tmp);
  if (cnt > 0)
    for (int t = t0; t < t1; ++t) {
      const unsigned long long k = sk[t];
      bool take = k > pref;
      if (!take && k == pref && take_eq > 0) {
        take = true;
        --take_eq;
      }
      if (take) out[pos++] = s_end + t;
    }
  if (tid == 0) *count = cnt;
}

// Attention selector, one layer: block (span row r, query head hh) writes the
// softmax over the pool of q_{r,hh} . K_layer[j] / sqrt(dh) into
// probs[(r*H + hh) * c + (j - s_end)].  dh * sizeof(T) is 128, 256 or 512
// bytes (dh 64 or 128), so a key row is 8, 16 or 32 lanes' 16-byte loads.
template <typename T>
__global__ void __launch_bounds__(256)
    k_attn_select_probs(const float *q, int H, int G, int dh, int layer, KVView v, int s_end,
                        int n, float *probs, float scale, int in_smem) {
  int r = blockIdx.x / H, hh = blockIdx.x % H, g = hh / (H / G);
  int c = n - s_end;
  extern __shared__ float qs[];
  __shared__ float red[32];
  for (int i = threadIdx.x; i < dh; i += blockDim.x)
    qs[i] = q[(size_t)r * H * dh + (size_t)hh * dh + i];
  __syncthreads();
  const T *kc = (const T *)v.pages;
  float *pr = probs + (size_t)blockIdx.x * c;
  // the row's logits: in shared memory after q when they fit (one write of
  // the probabilities to global at the end), else in place in probs
  float *buf = in_smem ? qs + dh : pr;
  float mx = -INFINITY;
  // L lanes read one key row with 16-byte loads (a contiguous row per group
  // of lanes, so a warp's load is L-way coalesced) and combine their partial
  // dot products by shuffles: blockDim / L keys per iteration
  constexpr int EPV = 16 / (int)sizeof(T);  // elements per 16-byte load
  const int L = dh / EPV;                   // 8, 16 or 32 lanes (dh 64 or 128)
  const int sub = threadIdx.x % L, kk = threadIdx.x / L, kpi = blockDim.x / L;
  const float *qv = qs + sub * EPV;
  constexpr int U = 8;  // keys per lane group in flight: U loads issued before any use
  for (int t0 = 0; t0 < c; t0 += kpi * U) {
    uint4 raw[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int t = t0 + u * kpi + kk;
      raw[u] = t < c ? *(const uint4 *)(kc + v.offset(layer, 0, g, s_end + t) + sub * EPV)
                     : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int t = t0 + u * kpi + kk;
      float s = 0.f;
      if constexpr (sizeof(T) == 2) {
        const __nv_bfloat162 *b = (const __nv_bfloat162 *)&raw[u];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(b[e]);
          s += qv[2 * e] * f.x;
          s += qv[2 * e + 1] * f.y;
        }
      } else {
        const float *f = (const float *)&raw[u];
#pragma unroll
        for (int e = 0; e < 4; ++e) s += qv[e] * f[e];
      }
      for (int off = L >> 1; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
      if (t < c && sub == 0) {
        s *= scale;
        buf[t] = s;
        mx = fmaxf(mx, s);
      }
    }
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
    float e = expf(buf[t] - mx);
    buf[t] = e;
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
  for (int t = threadIdx.x; t < c; t += blockDim.x) pr[t] = buf[t] * inv;
}

// score[j] += sum over (row, head) of probs, in a fixed order: a CTA takes 32
// keys; its 8 warps sum interleaved slices of the RH rows (coalesced along the
// keys), then warp 0 adds the 8 slice sums in slice order.
constexpr int ACC_SLICES = 8;
__global__ void __launch_bounds__(32 * ACC_SLICES)
    k_attn_select_accum(const float *probs, int RH, int c, int s_end, float *score) {
  __shared__ float part[ACC_SLICES][32];
  const int kk = threadIdx.x & 31, sl = threadIdx.x >> 5;
  const int t = blockIdx.x * 32 + kk;
  float s = 0.f;
  if (t < c) {
#pragma unroll 8
    for (int rh = sl; rh < RH; rh += ACC_SLICES) s += probs[(size_t)rh * c + t];
  }
  part[sl][kk] = s;
  __syncthreads();
  if (sl == 0 && t < c) {
    float tot = 0.f;
#pragma unroll
    for (int i = 0; i < ACC_SLICES; ++i) tot += part[i][kk];
    score[s_end + t] += tot;
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
  size_t smem = (size_t)c * sizeof(unsigned long long);
  if (smem >= 32 * 1024) {  // the default 48 KB limit also covers static shared memory
    cudaError_t e = cudaFuncSetAttribute(k_topk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cudaGetErrorString(e);
  }
  k_topk<<<1, TOPK_THREADS, smem, s>>>(keys, c, s_end, K, nonzero_only, out, count);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

void launch_attn_select_scores(const float *q, int S, const Dims &dm, int layer, KVView v,
                               int s_end, int n, float *probs_ws, float *scores, cudaStream_t s) {
  int c = n - s_end;
  if (c <= 0 || S <= 0) return;
  float scale = (float)(1.0 / sqrt((double)dm.dh));
  // q, then the row's logits when both fit the default 48 KB of shared memory
  const size_t with_row = (size_t)(dm.dh + c) * sizeof(float);
  const int in_smem = with_row <= (48u << 10) ? 1 : 0;
  const size_t smem = in_smem ? with_row : (size_t)dm.dh * sizeof(float);
  if (dm.dtype == KVR_DTYPE_BF16)
    k_attn_select_probs<__nv_bfloat16><<<S * dm.H, 256, smem, s>>>(
        q, dm.H, dm.G, dm.dh, layer, v, s_end, n, probs_ws, scale, in_smem);
  else
    k_attn_select_probs<float><<<S * dm.H, 256, smem, s>>>(q, dm.H, dm.G, dm.dh, layer, v, s_end,
                                                            n, probs_ws, scale, in_smem);
  k_attn_select_accum<<<(c + 31) / 32, 32 * ACC_SLICES, 0, s>>>(probs_ws, S * dm.H, c, s_end,
                                                                  scores);
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
