// k_rows.cu -- per-row kernels of the repair pass: seeded weight init,
// embedding gather, RMSNorm, RoPE + K/V scatter into the paged cache,
// SwiGLU, and cache row readback / save / restore.
#include "kvr_internal.cuh"

namespace kvr {

namespace {

constexpr uint64_t GAMMA = 0x9E3779B97F4A7C15ull;

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

template <typename T>
__device__ __forceinline__ float ld(const T *p, size_t i);
template <>
__device__ __forceinline__ float ld<float>(const float *p, size_t i) { return p[i]; }
template <>
__device__ __forceinline__ float ld<__nv_bfloat16>(const __nv_bfloat16 *p, size_t i) {
  return __bfloat162float(p[i]);
}

template <typename T>
__device__ __forceinline__ void st(T *p, size_t i, float v);
template <>
__device__ __forceinline__ void st<float>(float *p, size_t i, float v) { p[i] = v; }
template <>
__device__ __forceinline__ void st<__nv_bfloat16>(__nv_bfloat16 *p, size_t i, float v) {
  p[i] = __float2bfloat16_rn(v);
}

// One element of the seeded weight definition (SplitMix64 stream, Irwin-Hall
// sum of four 16-bit lanes, scaled in double, rounded to fp32).
__device__ __forceinline__ float init_value(uint64_t tseed, int64_t e, double scale) {
  uint64_t r = mix64(tseed + (uint64_t)(e + 1) * GAMMA);
  int s = (int)(r & 0xFFFF) + (int)((r >> 16) & 0xFFFF) + (int)((r >> 32) & 0xFFFF) +
          (int)(r >> 48);
  double x = (double)(s - 2 * 65535) * scale;
  return __double2float_rn(x);
}

__global__ void k_init_tensor(void *dst, int dtype, int out_f32, uint64_t tseed, double scale,
                              int64_t rows, int64_t cols, int64_t row_off, int inter) {
  int64_t total = rows * cols;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    float f = init_value(tseed, e, scale);
    int64_t r = e / cols, c = e % cols;
    int64_t dr = inter == 0 ? row_off + r
                            : (r / GU_BLOCK) * (2 * GU_BLOCK) + (inter == 2 ? GU_BLOCK : 0) +
                                  r % GU_BLOCK;
    size_t o = (size_t)(dr * cols + c);
    if (dtype == KVR_DTYPE_BF16) {
      __nv_bfloat16 b = __float2bfloat16_rn(f);
      if (out_f32)
        ((float *)dst)[o] = __bfloat162float(b);
      else
        ((__nv_bfloat16 *)dst)[o] = b;
    } else {
      ((float *)dst)[o] = f;
    }
  }
}

__global__ void k_fill_f32(float *dst, float v, size_t n) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x)
    dst[i] = v;
}

template <typename T>
__global__ void k_embed_rows(const T *embed, const int32_t *tokens,
                             const int32_t *const *doc_tokens, const int32_t *rowdoc,
                             const int32_t *pos, int d, float *h) {
  TraceScope ts(TK_EMBED);
  pdl_trigger();
  pdl_wait();
  ts.waited();
  int i = blockIdx.x;
  const int32_t *tk = doc_tokens ? doc_tokens[rowdoc[i]] : tokens;
  size_t base = (size_t)tk[pos[i]] * d;
  for (int c = threadIdx.x; c < d; c += blockDim.x) h[(size_t)i * d + c] = ld(embed, base + c);
}

// One block per row (d <= 8192, d % 4 == 0), each load issued before its
// first use: 1024 threads with NV = 1 float4 each up to d = 4096 (else 2)
// for a pass of a few rows, 256 threads with NV = d / 1024 for many.  Block i
// normalises h row row0 + i into out row i.  With a split view, the row is
// first completed from the GEMM's split-tile partials (their tile table is
// built once per block in shared memory) and written back to h.
constexpr int NORM_THREADS = 1024;   // a few rows: one float4 per thread, one round trip
constexpr int NORM_THREADS_WIDE = 256;  // many rows: several CTAs per SM, fewer waves
// The wide variant asks for four CTAs per SM: at 86 registers only two fit
// (prefill norms 3.2 against 2.9 ms).
template <typename T, int NV, int TPB>
__global__ void __launch_bounds__(TPB, TPB == NORM_THREADS_WIDE && NV <= 4 ? 4 : 1)
    k_rmsnorm(float *h, const float *g, int row0, int d, float eps, T *out, const SplitView sv) {
  __shared__ SplitTile tiles[64];
  __shared__ float red[TPB / 32];
  TraceScope ts(TK_NORM);
  pdl_trigger();
  const int i = blockIdx.x, row = row0 + i;
  const int nq = d >> 2;
  if (sv.ws && (int)threadIdx.x < (d >> 7)) {
    const int mt = row / sv.BN;
    tiles[threadIdx.x] = split_tile(sv, (long long)threadIdx.x * sv.m_tiles + mt);
  }
  // the gains are weights: read them before waiting on the residual's producer
  float4 gw[NV];
#pragma unroll
  for (int k = 0; k < NV; ++k) {
    const int q = k * TPB + threadIdx.x;
    gw[k] = q < nq ? ((const float4 *)g)[q] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  pdl_wait();
  ts.waited();
  if (sv.ws) __syncthreads();
  float4 *x = (float4 *)(h + (size_t)row * d);
  float4 v[NV];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < NV; ++k) {
    const int q = k * TPB + threadIdx.x;
    v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (q < nq) {
      v[k] = x[q];
      if (sv.ws) {
        const SplitTile st = tiles[q >> 5];
        if (st.i0 != st.i1) {
          v[k] = split_value4(sv, st, v[k], row, 4 * q);
          x[q] = v[k];
        }
      }
    }
    ss += v[k].x * v[k].x + v[k].y * v[k].y + v[k].z * v[k].z + v[k].w * v[k].w;
  }
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < TPB / 32; ++w) tot += red[w];
  const float r = 1.0f / sqrtf(tot / (float)d + eps);
#pragma unroll
  for (int k = 0; k < NV; ++k) {
    const int q = k * TPB + threadIdx.x;
    if (q < nq) {
      const float4 w = gw[k];
      const size_t o = (size_t)i * d + 4 * q;
      st(out, o, v[k].x * r * w.x);
      st(out, o + 1, v[k].y * r * w.y);
      st(out, o + 2, v[k].z * r * w.z);
      st(out, o + 3, v[k].w * r * w.w);
    }
  }
}

// grid (ceil(M / rpb), ceil((H + 2G) / ROPE_HEADS)), block ROPE_HEADS * dh/2:
// rotate q and k heads at the row's position; q -> q_out fp32 (if given) and
// qb_out, k and v -> cache (if write_kv) and rows_out (if given).  With a
// split view the projection is completed from the GEMM's split-tile
// partials.  Positions, the RoPE table, the page table and the bias are
// written before the pass, so they are read before the wait on the
// projection.  RPB > 1 (a prefill chunk, no split view): the CTA's RPB rows
// are loaded together, one round trip for all of them.
constexpr int ROPE_HEADS = 8;  // heads per CTA
constexpr int ROPE_RPB = 8;    // rows per CTA of a many-row pass
template <typename T, int RPB>
__global__ void k_rope_scatter(const float *qkv, const float2 *rope, const int32_t *pos, int M,
                               int rpb, int H, int G, int dh, int layer, const KVView *views,
                               const int32_t *rowdoc, KVView single, float *q_out,
                               __nv_bfloat16 *qb_out, float qscale, int write_kv,
                               const SplitView sv, T *rows_out, int L) {
  TraceScope ts(TK_ROPE);
  pdl_trigger();
  const int half = dh >> 1;
  const int hh = blockIdx.y * ROPE_HEADS + threadIdx.x / half, t = threadIdx.x % half;
  if (hh >= H + 2 * G) return;
  const int Nqkv = (H + 2 * G) * dh;
  const int n1 = hh * dh + t, n2 = n1 + half;
  const int kv = hh < H + G ? 0 : 1, gk = hh - H - kv * G;
  // the row's cache entry (o) and rows_out entry (ro), for k and v heads
  auto kv_dst = [&](int i, int p, T *&c, size_t &o, size_t &ro) {
    c = nullptr;
    if (hh >= H && write_kv) {
      const KVView v = views ? views[rowdoc[i]] : single;
      c = (T *)v.pages;
      o = v.offset(layer, kv, gk, p);
      // rows_out: K then V, each [M][L][G][dh]
      ro = ((((size_t)kv * M + i) * L + layer) * G + gk) * dh;
    }
  };
  auto out = [&](int i, float x1, float x2, float2 cs, T *c, size_t o, size_t ro) {
    if (hh < H + G) {
      const float r1r = x1 * cs.x - x2 * cs.y;
      const float r2r = x2 * cs.x + x1 * cs.y;
      x1 = r1r;
      x2 = r2r;
    }
    if (hh < H) {
      if (q_out) {
        float *qo = q_out + (size_t)i * H * dh + (size_t)hh * dh;
        qo[t] = x1;
        qo[t + half] = x2;
      }
      if (qb_out) {
        __nv_bfloat16 *qb = qb_out + (size_t)i * H * dh + (size_t)hh * dh;
        qb[t] = __float2bfloat16_rn(x1 * qscale);
        qb[t + half] = __float2bfloat16_rn(x2 * qscale);
      }
      return;
    }
    if (!c) return;
    st(c, o + t, x1);
    st(c, o + t + half, x2);
    if (rows_out) {
      st(rows_out, ro + t, x1);
      st(rows_out, ro + t + half, x2);
    }
  };
  if constexpr (RPB > 1) {
    const int r0 = blockIdx.x * RPB, nr = min(RPB, M - r0);
    int p[RPB];
    float2 cs[RPB];
    T *c[RPB];
    size_t o[RPB], ro[RPB];
#pragma unroll
    for (int k = 0; k < RPB; ++k) {
      p[k] = k < nr ? pos[r0 + k] : 0;
      cs[k] = hh < H + G && k < nr ? rope[(size_t)p[k] * half + t] : make_float2(1.f, 0.f);
      c[k] = nullptr;
      if (k < nr) kv_dst(r0 + k, p[k], c[k], o[k], ro[k]);
    }
    pdl_wait();
    ts.waited();
    float x1[RPB], x2[RPB];
#pragma unroll
    for (int k = 0; k < RPB; ++k) {
      const float *x = qkv + (size_t)(r0 + k) * Nqkv;
      x1[k] = k < nr ? x[n1] : 0.f;
      x2[k] = k < nr ? x[n2] : 0.f;
    }
#pragma unroll
    for (int k = 0; k < RPB; ++k)
      if (k < nr) out(r0 + k, x1[k], x2[k], cs[k], c[k], o[k], ro[k]);
    return;
  }
  // rows r0 .. r1-1 one after another; the first row's position, table
  // entries and split tile are read before the wait
  const int r0 = blockIdx.x * rpb, r1 = min(M, r0 + rpb);
  for (int i = r0; i < r1; ++i) {
    const int p = pos[i];
    float2 cs = make_float2(1.f, 0.f);
    if (hh < H + G) cs = rope[(size_t)p * half + t];
    T *c;
    size_t o = 0, ro = 0;
    kv_dst(i, p, c, o, ro);
    // dh divides 128: both halves of the head lie in one feature tile
    SplitTile stl{0, 0, 0};
    float b1 = 0.f, b2 = 0.f;
    if (sv.ws) {
      stl = split_tile(sv, (long long)((hh * dh) >> 7) * sv.m_tiles + i / sv.BN);
      if (sv.bias) {
        b1 = sv.bias[n1];
        b2 = sv.bias[n2];
      }
    }
    const bool split = sv.ws && stl.i0 != stl.i1;
    if (i == r0) {
      pdl_wait();
      ts.waited();
    }
    float x1, x2;
    if (split) {
      const size_t off = (size_t)(i - (i / sv.BN) * sv.BN) * 128;
      x1 = b1 + split_sum(sv, stl, off + (n1 & 127));
      x2 = b2 + split_sum(sv, stl, off + (n2 & 127));
    } else {
      const float *x = qkv + (size_t)i * Nqkv;
      x1 = x[n1];
      x2 = x[n2];
    }
    out(i, x1, x2, cs, c, o, ro);
  }
}

template <typename T>
__global__ void k_swiglu(const float *gu, int M, int F, T *act) {
  size_t total = (size_t)M * F;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total;
       e += (size_t)gridDim.x * blockDim.x) {
    size_t m = e / F;
    int f = (int)(e % F);
    size_t base = m * 2 * F + (size_t)(f / GU_BLOCK) * 2 * GU_BLOCK + f % GU_BLOCK;
    float g = gu[base], u = gu[base + GU_BLOCK];
    st(act, e, g / (1.0f + expf(-g)) * u);
  }
}

template <typename T>
__global__ void k_cache_gather(KVView v, const int32_t *pos, int n_pos, int l0, int nl, int G,
                               int dh, float *k_out, float *v_out) {
  size_t total = (size_t)n_pos * nl * G * dh;
  const T *c = (const T *)v.pages;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total;
       e += (size_t)gridDim.x * blockDim.x) {
    int i = (int)(e % dh);
    size_t r = e / dh;
    int g = (int)(r % G);
    r /= G;
    int l = (int)(r % nl);
    int p = (int)(r / nl);
    k_out[e] = ld(c, v.offset(l0 + l, 0, g, pos[p]) + i);
    v_out[e] = ld(c, v.offset(l0 + l, 1, g, pos[p]) + i);
  }
}

// K/V of the given positions, layers l0 .. l0+nl-1, as stored: 16-byte
// pieces of the cache rows (a row is head_dim elements, a multiple of 16
// bytes), vr pieces a row, output [n_pos][nl][G][row].
__global__ void k_cache_gather_raw(KVView v, const int32_t *pos, int n_pos, int l0, int nl, int G,
                                   int vr, int es, uint4 *k_out, uint4 *v_out) {
  const unsigned total = (unsigned)n_pos * nl * G * vr;
  const uint4 *c = (const uint4 *)v.pages;
  for (unsigned e = blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += gridDim.x * blockDim.x) {
    const unsigned i = e % vr;
    unsigned r = e / vr;
    const int g = (int)(r % G);
    r /= G;
    const int l = (int)(r % nl);
    const int p = pos[r / nl];
    k_out[e] = c[v.offset(l0 + l, 0, g, p) * es / 16 + i];
    v_out[e] = c[v.offset(l0 + l, 1, g, p) * es / 16 + i];
  }
}

// The inverse of k_cache_gather_raw for consecutive positions p0 .. p0+n_pos-1
// and every layer: rows [n_pos][L][G][dh] of k_in / v_in written into the pages.
template <typename T>
__global__ void k_cache_scatter_raw(KVView v, int p0, int n_pos, const T *k_in, const T *v_in) {
  const int L = v.L, G = v.G, dh = v.dh;
  size_t total = (size_t)n_pos * L * G * dh;
  T *c = (T *)v.pages;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total;
       e += (size_t)gridDim.x * blockDim.x) {
    int i = (int)(e % dh);
    size_t r = e / dh;
    int g = (int)(r % G);
    r /= G;
    int l = (int)(r % L);
    int p = p0 + (int)(r / L);
    c[v.offset(l, 0, g, p) + i] = k_in[e];
    c[v.offset(l, 1, g, p) + i] = v_in[e];
  }
}

// buf layout [n_pos][nl][2][G][dh] in the cache dtype
template <typename T>
__global__ void k_rows_copy(KVView v, const int32_t *pos, int n_pos, int l0, int nl, T *buf,
                            int to_buf) {
  int G = v.G, dh = v.dh;
  size_t total = (size_t)n_pos * nl * 2 * G * dh;
  T *c = (T *)v.pages;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total;
       e += (size_t)gridDim.x * blockDim.x) {
    int i = (int)(e % dh);
    size_t r = e / dh;
    int g = (int)(r % G);
    r /= G;
    int kv = (int)(r % 2);
    r /= 2;
    int l = (int)(r % nl);
    int p = (int)(r / nl);
    size_t o = v.offset(l0 + l, kv, g, pos[p]) + i;
    if (to_buf)
      buf[e] = c[o];
    else
      c[o] = buf[e];
  }
}

// Transplant: copy K/V of every layer at the listed positions from one
// document's pages into another's (same model shape).
template <typename T>
__global__ void k_transplant(KVView dst, KVView src, const int32_t *pos, int n_pos) {
  const int L = dst.L, G = dst.G, dh = dst.dh;
  size_t total = (size_t)n_pos * L * 2 * G * dh;
  const T *s = (const T *)src.pages;
  T *d = (T *)dst.pages;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total;
       e += (size_t)gridDim.x * blockDim.x) {
    int i = (int)(e % dh);
    size_t r = e / dh;
    int g = (int)(r % G);
    r /= G;
    int kv = (int)(r % 2);
    r /= 2;
    int l = (int)(r % L);
    int p = pos[r / L];
    d[dst.offset(l, kv, g, p) + i] = s[src.offset(l, kv, g, p) + i];
  }
}

// out[i] = logits[i][target[i]] - logsumexp(logits[i]) for each row.
__global__ void __launch_bounds__(256) k_row_logprob(const float *logits, int V,
                                                     const int32_t *target, float *out) {
  const float *x = logits + (size_t)blockIdx.x * V;
  __shared__ float red[8];
  float mx = -INFINITY;
  for (int j = threadIdx.x; j < V; j += 256) mx = fmaxf(mx, x[j]);
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  __syncthreads();
  mx = red[0];
  for (int w = 1; w < 8; ++w) mx = fmaxf(mx, red[w]);
  __syncthreads();
  float sm = 0.f;
  for (int j = threadIdx.x; j < V; j += 256) sm += expf(x[j] - mx);
  for (int o = 16; o > 0; o >>= 1) sm += __shfl_xor_sync(0xffffffffu, sm, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sm;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += red[w];
    out[blockIdx.x] = x[target[blockIdx.x]] - (mx + logf(t));
  }
}

int grid_for(size_t n, int block) {
  size_t g = (n + block - 1) / block;
  return (int)(g > 65535 * 8 ? 65535 * 8 : (g == 0 ? 1 : g));
}

}  // namespace

void launch_init_tensor(void *dst, int dtype, bool out_f32, uint64_t tseed, double scale,
                        int64_t rows, int64_t cols, int64_t row_off, int interleave,
                        cudaStream_t s) {
  size_t n = (size_t)(rows * cols);
  k_init_tensor<<<grid_for(n, 256), 256, 0, s>>>(dst, dtype, out_f32 ? 1 : 0, tseed, scale, rows,
                                                  cols, row_off, interleave);
}

void launch_fill_f32(float *dst, float v, size_t n, cudaStream_t s) {
  k_fill_f32<<<grid_for(n, 256), 256, 0, s>>>(dst, v, n);
}

void launch_embed_rows(const void *embed, int dtype, const int32_t *tokens,
                       const int32_t *const *doc_tokens, const int32_t *rowdoc,
                       const int32_t *pos, int M, int d, float *h, cudaStream_t s) {
  if (M <= 0) return;
  if (dtype == KVR_DTYPE_BF16)
    launch_pdl(k_embed_rows<__nv_bfloat16>, M, 256, 0, s, (const __nv_bfloat16 *)embed, tokens,
               doc_tokens, rowdoc, pos, d, h);
  else
    launch_pdl(k_embed_rows<float>, M, 256, 0, s, (const float *)embed, tokens, doc_tokens,
               rowdoc, pos, d, h);
}

void launch_rmsnorm(float *h, const float *g, int row0, int M, int d, double eps, void *out,
                    int out_dtype, cudaStream_t s, const SplitView *sv) {
  if (M <= 0) return;
  const SplitView v = sv ? *sv : SplitView{};
  // A pass of a few rows is latency-bound: 1024 threads, each with one
  // float4 in flight.  Hundreds of rows (prefill) run in waves: 256 threads a
  // row, several rows per SM at once.
  if (M > 256 && d <= 4 * 8 * NORM_THREADS_WIDE) {
    constexpr int W = NORM_THREADS_WIDE;
    const int nv = (d + 4 * W - 1) / (4 * W);
    if (out_dtype == KVR_DTYPE_BF16) {
      auto k = nv <= 1 ? k_rmsnorm<__nv_bfloat16, 1, W>
               : nv <= 2 ? k_rmsnorm<__nv_bfloat16, 2, W>
               : nv <= 4 ? k_rmsnorm<__nv_bfloat16, 4, W>
                         : k_rmsnorm<__nv_bfloat16, 8, W>;
      launch_pdl(k, M, W, 0, s, h, g, row0, d, (float)eps, (__nv_bfloat16 *)out, v);
    } else {
      auto k = nv <= 1 ? k_rmsnorm<float, 1, W>
               : nv <= 2 ? k_rmsnorm<float, 2, W>
               : nv <= 4 ? k_rmsnorm<float, 4, W>
                         : k_rmsnorm<float, 8, W>;
      launch_pdl(k, M, W, 0, s, h, g, row0, d, (float)eps, (float *)out, v);
    }
    return;
  }
  const bool one = d <= 4 * NORM_THREADS;
  if (out_dtype == KVR_DTYPE_BF16)
    launch_pdl(one ? k_rmsnorm<__nv_bfloat16, 1, NORM_THREADS>
                   : k_rmsnorm<__nv_bfloat16, 2, NORM_THREADS>,
               M, NORM_THREADS, 0, s, h, g, row0, d, (float)eps, (__nv_bfloat16 *)out, v);
  else
    launch_pdl(one ? k_rmsnorm<float, 1, NORM_THREADS> : k_rmsnorm<float, 2, NORM_THREADS>, M,
               NORM_THREADS, 0, s, h, g, row0, d, (float)eps, (float *)out, v);
}

void launch_rope_scatter(const float *qkv, const float2 *rope, const int32_t *pos, int M,
                         const Dims &dm, int layer, const KVView *views, const int32_t *rowdoc,
                         KVView single, float *q_out, void *qb_out, float qscale, bool write_kv,
                         cudaStream_t s, const SplitView *sv, void *rows_out) {
  if (M <= 0) return;
  const SplitView v = sv ? *sv : SplitView{};
  // a prefill chunk: several rows per CTA (one row per CTA spent its time
  // starting CTAs), loaded together when the projection is complete
  const int rpb = M >= 1024 ? ROPE_RPB : 1;
  const bool batched = rpb > 1 && !v.ws;
  dim3 grid((M + rpb - 1) / rpb, (dm.H + 2 * dm.G + ROPE_HEADS - 1) / ROPE_HEADS);
  const int threads = ROPE_HEADS * dm.dh / 2;
  int wk = write_kv ? 1 : 0;
  auto go = [&](auto *tag) {
    using T = std::remove_pointer_t<decltype(tag)>;
    launch_pdl(batched ? k_rope_scatter<T, ROPE_RPB> : k_rope_scatter<T, 1>, grid, threads, 0, s,
               qkv, rope, pos, M, rpb, dm.H, dm.G, dm.dh, layer, views, rowdoc, single, q_out,
               (__nv_bfloat16 *)qb_out, qscale, wk, v, (T *)rows_out, dm.L);
  };
  if (dm.dtype == KVR_DTYPE_BF16)
    go((__nv_bfloat16 *)nullptr);
  else
    go((float *)nullptr);
}

void launch_swiglu(const float *gu, int M, int F, void *act, int dtype, cudaStream_t s) {
  if (M <= 0) return;
  size_t n = (size_t)M * F;
  if (dtype == KVR_DTYPE_BF16)
    k_swiglu<<<grid_for(n, 256), 256, 0, s>>>(gu, M, F, (__nv_bfloat16 *)act);
  else
    k_swiglu<<<grid_for(n, 256), 256, 0, s>>>(gu, M, F, (float *)act);
}

void launch_cache_gather(KVView v, int dtype, const int32_t *pos, int n_pos, int l0, int l1,
                         int G, int dh, float *k_out, float *v_out, cudaStream_t s) {
  size_t n = (size_t)n_pos * (l1 - l0) * G * dh;
  if (n == 0) return;
  if (dtype == KVR_DTYPE_BF16)
    k_cache_gather<__nv_bfloat16><<<grid_for(n, 256), 256, 0, s>>>(v, pos, n_pos, l0, l1 - l0, G,
                                                                    dh, k_out, v_out);
  else
    k_cache_gather<float><<<grid_for(n, 256), 256, 0, s>>>(v, pos, n_pos, l0, l1 - l0, G, dh,
                                                            k_out, v_out);
}

void launch_cache_gather_raw(KVView v, int dtype, const int32_t *pos, int n_pos, int l0, int l1,
                             int G, int dh, void *k_out, void *v_out, cudaStream_t s) {
  const int es = dtype == KVR_DTYPE_BF16 ? 2 : 4, vr = dh * es / 16;
  const size_t per_pos = (size_t)(l1 - l0) * G * vr;
  if (per_pos == 0) return;
  // launches of fewer than 2^31 pieces (the kernel indexes in 32 bits)
  const int chunk = (int)std::min<size_t>((size_t)n_pos, ((size_t)1 << 31) / per_pos);
  for (int p0 = 0; p0 < n_pos; p0 += chunk) {
    const int np = std::min(chunk, n_pos - p0);
    k_cache_gather_raw<<<grid_for(np * per_pos, 256), 256, 0, s>>>(
        v, pos + p0, np, l0, l1 - l0, G, vr, es, (uint4 *)k_out + p0 * per_pos,
        (uint4 *)v_out + p0 * per_pos);
  }
}

void launch_cache_scatter_raw(KVView v, int dtype, int p0, int n_pos, const void *k_in,
                              const void *v_in, cudaStream_t s) {
  size_t n = (size_t)n_pos * v.L * v.G * v.dh;
  if (n == 0) return;
  if (dtype == KVR_DTYPE_BF16)
    k_cache_scatter_raw<__nv_bfloat16><<<grid_for(n, 256), 256, 0, s>>>(
        v, p0, n_pos, (const __nv_bfloat16 *)k_in, (const __nv_bfloat16 *)v_in);
  else
    k_cache_scatter_raw<float><<<grid_for(n, 256), 256, 0, s>>>(v, p0, n_pos, (const float *)k_in,
                                                                 (const float *)v_in);
}

void launch_transplant(KVView dst, KVView src, int dtype, const int32_t *pos, int n_pos,
                       cudaStream_t s) {
  size_t n = (size_t)n_pos * dst.L * 2 * dst.G * dst.dh;
  if (n == 0) return;
  if (dtype == KVR_DTYPE_BF16)
    k_transplant<__nv_bfloat16><<<grid_for(n, 256), 256, 0, s>>>(dst, src, pos, n_pos);
  else
    k_transplant<float><<<grid_for(n, 256), 256, 0, s>>>(dst, src, pos, n_pos);
}

void launch_row_logprob(const float *logits, int rows, int V, const int32_t *target, float *out,
                        cudaStream_t s) {
  if (rows > 0) k_row_logprob<<<rows, 256, 0, s>>>(logits, V, target, out);
}

void launch_rows_copy(KVView v, int dtype, const int32_t *pos, int n_pos, int l0, int l1,
                      void *buf, bool to_buf, cudaStream_t s) {
  size_t n = (size_t)n_pos * (l1 - l0) * 2 * v.G * v.dh;
  if (n == 0) return;
  if (dtype == KVR_DTYPE_BF16)
    k_rows_copy<<<grid_for(n, 256), 256, 0, s>>>(v, pos, n_pos, l0, l1 - l0,
                                                  (__nv_bfloat16 *)buf, to_buf ? 1 : 0);
  else
    k_rows_copy<<<grid_for(n, 256), 256, 0, s>>>(v, pos, n_pos, l0, l1 - l0, (float *)buf,
                                                  to_buf ? 1 : 0);
}

KVR_TRACE_ATTACH(trace_attach_rows)

}  // namespace kvr
