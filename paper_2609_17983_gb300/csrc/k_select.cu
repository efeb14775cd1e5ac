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

// Key of pool entry t (position s_end + t) under a simple policy; bnd: the
// EditLocal@boundary boundary.
__device__ __forceinline__ unsigned long long simple_key(const SimpleKeys &g, int s_end, int t,
                                                        int bnd) {
  const int j = s_end + t;
  if (g.policy == KVR_POLICY_RANDOM) {
    // first SplitMix64 output of state seed ^ (j * gamma)
    return mix64((g.seed ^ ((uint64_t)j * GAMMA)) + GAMMA);
  }
  // nearest to the span first
  unsigned long long k = 0x100000000ull - (unsigned long long)t;
  if (g.policy == KVR_POLICY_STRUCTURAL && g.tokens[j] != g.delim) k = 0;
  if (g.policy == KVR_POLICY_EDITLOCAL_BOUNDARY && j > bnd) k = 0;
  return k;
}

__global__ void k_float_keys(const float *scores, int n, int s_end, unsigned long long *keys) {
  int c = n - s_end;
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < c; t += gridDim.x * blockDim.x)
    keys[t] = (unsigned long long)ord_f32(scores[s_end + t]) + 1ull;
}

// Top-K of c (key, index) pairs, one CTA of TOPK_THREADS: key descending, ties to
// the lowest index, the chosen indices written ascending.  Instead of a sort,
// the K-th key T is found by an MSB-first radix select (8 bits per pass, a
// shared-memory histogram of the keys that still match the prefix), starting
// at the highest 8-bit digit in which the keys differ (the AND and OR of all
// keys give the digits they share, which the passes would only confirm); then
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
           int32_t *out, int32_t *count, const SimpleKeys gen, const int *flag_in,
           int32_t *flag_out) {
  extern __shared__ unsigned long long sk[];  // c keys
  __shared__ int hist[256];
  __shared__ int scan_tmp[TOPK_THREADS / 32];
  __shared__ int s_elig, s_bin, s_above;
  __shared__ unsigned long long s_and, s_or;
  const int tid = threadIdx.x;
  if (gen.policy == KVR_POLICY_EDITLOCAL ||
      (gen.policy == KVR_POLICY_EDITLOCAL_BOUNDARY && nonzero_only)) {
    // EditLocal's keys fall strictly with t, all nonzero (@boundary: nonzero
    // up to the boundary, zero after it, and only nonzero keys eligible): the
    // K largest are the first K candidates, already in index order.
    const int avail = gen.policy == KVR_POLICY_EDITLOCAL ? c : min(c, *gen.bound - s_end + 1);
    const int cnt = min(K, max(avail, 0));
    for (int t = tid; t < cnt; t += TOPK_THREADS) out[t] = s_end + t;
    if (tid == 0) {
      *count = cnt;
      if (flag_in) *flag_out = *flag_in;
    }
    return;
  }
  const int E = (c + TOPK_THREADS - 1) / TOPK_THREADS;
  const int t0 = min(c, tid * E), t1 = min(c, t0 + E);
  if (tid == 0) {
    s_elig = 0;
    s_and = ~0ull;
    s_or = 0ull;
  }
  __syncthreads();
  const int bnd = gen.policy == KVR_POLICY_EDITLOCAL_BOUNDARY ? *gen.bound : 0;
  int local = 0;
  unsigned long long kand = ~0ull, kor = 0ull;
  for (int t = tid; t < c; t += TOPK_THREADS) {
    const unsigned long long k = gen.policy >= 0 ? simple_key(gen, s_end, t, bnd) : keys[t];
    sk[t] = k;
    kand &= k;
    kor |= k;
    local += (!nonzero_only || k != 0ull) ? 1 : 0;
  }
  for (int o = 16; o > 0; o >>= 1) {
    local += __shfl_xor_sync(0xffffffffu, local, o);
    kand &= __shfl_xor_sync(0xffffffffu, kand, o);
    kor |= __shfl_xor_sync(0xffffffffu, kor, o);
  }
  if ((tid & 31) == 0) {
    atomicAdd(&s_elig, local);
    atomicAnd(&s_and, kand);
    atomicOr(&s_or, kor);
  }
  __syncthreads();
  const int cnt = min(K, s_elig);
  // radix select: prefix/mask of T, need = how many keys equal to the prefix
  // (so far) are still to be taken.  The digits above dtop are the same in
  // every key: they start the prefix.
  const unsigned long long differ = s_or ^ s_and;
  const int dtop = differ ? (63 - __clzll((long long)differ)) / 8 * 8 : -8;
  unsigned long long mask = dtop >= 56 ? 0ull : ~0ull << (dtop + 8);
  unsigned long long pref = s_and & mask;
  int need = cnt;
  for (int d = dtop; d >= 0 && need > 0; d -= 8) {
    for (int i = tid; i < 256; i += TOPK_THREADS) hist[i] = 0;
    __syncthreads();
    // lanes whose keys fall in the same bin add their count once: keys near
    // the span (EditLocal) share their upper digits, and one shared-memory
    // address taking every key serialises the pass
    for (int e = 0; e < E; ++e) {
      const int t = t0 + e;
      const unsigned long long k = t < t1 ? sk[t] : 0ull;
      const int bin = t < t1 && (k & mask) == pref ? (int)(k >> d) & 255 : -1;
      const unsigned peers = __match_any_sync(0xffffffffu, bin);
      if (bin >= 0 && (tid & 31) == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
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
  if (tid == 0) {
    *count = cnt;
    if (flag_in) *flag_out = *flag_in;
  }
}

// Attention selector, one layer, in two kernels over a workspace.  The
// queries of kv group g are the span rows' heads hh with hh / (H/G) == g;
// within the group a query is ql = r * (H/G) + (hh mod H/G), globally
// qg = g * S * (H/G) + ql.  A CTA of k_attn_select_logits takes SEL_KC pool
// keys and SEL_QT queries of one group: the keys are read once into shared
// memory and serve every query of the tile (so a group's key rows leave L2
// once per query tile, not once per query).  It stores the scaled logits,
// logit[qg * c + (j - s_end)], and per query the chunk's max and sum of
// exp(logit - max); the last CTA of (group, query tile) to finish folds the
// chunk statistics into the pool softmax's max and 1 / sum.  Arrival is an
// atomic count with no waiting: every other CTA just exits.  The contraction
// runs on mma.sync for bf16 caches and on FFMA micro-tiles for fp32 caches.
constexpr int SEL_KC = 64, SEL_QT = 32, SEL_THREADS = 128;
constexpr int SEL_KG = SEL_KC / 4;   // fp32 path: key groups of 4 (a thread: 4 queries x 4 keys)
constexpr int SEL_LTS = SEL_KC + 4;  // logits tile row stride (floats)
constexpr int SEL_DH_MAX = 128;      // head_dim is 64 or 128 (checked at model creation)
constexpr int SEL_FOLD = 16;         // chunk statistics in flight per thread in the fold
static_assert(SEL_KG * (SEL_QT / 4) == SEL_THREADS, "one 4x4 micro-tile per thread");

struct SelWs {
  float *logit;  // [S*H][c]
  float2 *ml;    // [S*H][n_chunks] chunk (max, sum of exp)
  float2 *mz;    // [S*H] pool (max, 1 / sum of exp)
  int *cnt;      // [G][n_qtiles] arrivals
};

__host__ __device__ inline int sel_chunks(int c) { return (c + SEL_KC - 1) / SEL_KC; }

// (m, z) <- the (max, sum of exp) of the union of two sets, either possibly
// empty (m = -inf, z = 0).  Symmetric in its operands, bit for bit.
__device__ __forceinline__ void lse_merge(float &m, float &z, float m2, float z2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2, z = z2;
    return;
  }
  const float mm = fmaxf(m, m2);
  z = z * expf(m - mm) + z2 * expf(m2 - mm);
  m = mm;
}

__device__ __forceinline__ uint32_t bf2_bits(__nv_bfloat162 v) { return *(const uint32_t *)&v; }

// d[0..3] += A (16 x 16, row) . B (16 x 8, col), bf16 operands, fp32 accumulate
__device__ __forceinline__ void sel_mma_bf16(float *d, uint32_t a0, uint32_t a1, uint32_t a2,
                                             uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

template <typename T>
__global__ void __launch_bounds__(SEL_THREADS)
    k_attn_select_logits(const float *q, int S, int H, int G, int dh, int layer, KVView v,
                         int s_end, int c, float scale, SelWs ws) {
  TraceScope ts(TK_SELECT);
  pdl_trigger();
  const int chunk = blockIdx.x, g = blockIdx.y, qt = blockIdx.z, nch = gridDim.x;
  const int hpg = H / G, Nq = S * hpg;
  const int t0 = chunk * SEL_KC, q0 = qt * SEL_QT;
  const int nk = min(SEL_KC, c - t0), nq = min(SEL_QT, Nq - q0);
  const int tid = threadIdx.x;
  const size_t qg0 = (size_t)g * Nq + q0;
  extern __shared__ float4 sel_smem[];
  float *lt;  // [SEL_QT][SEL_LTS] logits, over the keys once they are consumed
  int *last;  // arrival flag, over the queries once they are consumed
  if constexpr (sizeof(T) == 2) {
    // bf16 keys: tensor cores (mma.sync m16n8k16, fp32 accumulate).  Each
    // query is split into two bf16 parts, q = q_hi + q_lo with q_lo the
    // rounding remainder, and logit = q_hi . k + q_lo . k: about 16 bits of
    // q's mantissa, the keys exact.  Rows are d-contiguous with a stride of
    // dh + 8 elements (4 mod 32 words), so a fragment load's 8 rows x 4
    // lanes fall on 32 banks.
    const int RS = dh + 8;
    __nv_bfloat16 *qh = (__nv_bfloat16 *)sel_smem;  // [SEL_QT][RS]
    __nv_bfloat16 *qo = qh + SEL_QT * RS;           // [SEL_QT][RS] the remainders
    __nv_bfloat16 *ks = qo + SEL_QT * RS;           // [SEL_KC][RS]
    lt = (float *)ks;
    last = (int *)qh;
    // the pool's stale keys: no kernel of the pass writes them, so they are
    // read before the wait on the predecessor; a thread issues all its loads
    // (page lookups, then rows) before it uses the first
    constexpr int KLD = SEL_KC * (SEL_DH_MAX / 8) / SEL_THREADS;
    const __nv_bfloat16 *kc = (const __nv_bfloat16 *)v.pages;
    const int L = dh / 8;  // 16-byte pieces per key row
    uint4 kx[KLD];
#pragma unroll
    for (int u = 0; u < KLD; ++u) {
      const int i = tid + u * SEL_THREADS, kk = i / L, sub = i % L;
      kx[u] = make_uint4(0u, 0u, 0u, 0u);
      if (kk < nk) kx[u] = *(const uint4 *)(kc + v.offset(layer, 0, g, s_end + t0 + kk) + sub * 8);
    }
#pragma unroll
    for (int u = 0; u < KLD; ++u) {
      const int i = tid + u * SEL_THREADS, kk = i / L, sub = i % L;
      if (kk < SEL_KC) *(uint4 *)(ks + kk * RS + sub * 8) = kx[u];  // rows of 16-byte multiples
    }
    pdl_wait();  // the queries come from the RoPE kernel just before
    ts.waited();
    constexpr int QLD = SEL_QT * (SEL_DH_MAX / 4) / SEL_THREADS;
    const int D4 = dh / 4;
    float4 qx[QLD];
#pragma unroll
    for (int u = 0; u < QLD; ++u) {
      const int i = tid + u * SEL_THREADS, ql = i / D4, d4 = i % D4;
      qx[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (ql < nq) {
        const int qq = q0 + ql, r = qq / hpg, hh = g * hpg + qq % hpg;
        qx[u] = *(const float4 *)(q + ((size_t)r * H + hh) * dh + 4 * d4);
      }
    }
#pragma unroll
    for (int u = 0; u < QLD; ++u) {
      const int i = tid + u * SEL_THREADS, ql = i / D4, d4 = i % D4;
      if (ql < SEL_QT) {
        const float2 x01 = make_float2(qx[u].x, qx[u].y), x23 = make_float2(qx[u].z, qx[u].w);
        const __nv_bfloat162 h01 = __float22bfloat162_rn(x01), h23 = __float22bfloat162_rn(x23);
        const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
        const __nv_bfloat162 l01 = __floats2bfloat162_rn(x01.x - f01.x, x01.y - f01.y);
        const __nv_bfloat162 l23 = __floats2bfloat162_rn(x23.x - f23.x, x23.y - f23.y);
        *(uint2 *)(qh + ql * RS + 4 * d4) = make_uint2(bf2_bits(h01), bf2_bits(h23));
        *(uint2 *)(qo + ql * RS + 4 * d4) = make_uint2(bf2_bits(l01), bf2_bits(l23));
      }
    }
    __syncthreads();
    if (tid == 0) trace_mark(0);  // keys and queries staged
    // warp w: keys 16w .. 16w + 15 (two n-tiles of 8), all SEL_QT queries
    // (two m-tiles of 16); lane: group gr = lane / 4, pair column gc
    const int warp = tid >> 5, lane = tid & 31, gr = lane >> 2, gc = (lane & 3) * 2;
    static_assert(SEL_QT == 32 && SEL_KC == 16 * (SEL_THREADS / 32), "warp tiling");
    float acc[2][2][4];
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[mt][nt][e] = 0.f;
    for (int k0 = 0; k0 < dh; k0 += 16) {
      uint32_t b[2][2];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        const __nv_bfloat16 *kr = ks + (16 * warp + 8 * nt + gr) * RS + k0 + gc;
        b[nt][0] = *(const uint32_t *)kr;
        b[nt][1] = *(const uint32_t *)(kr + 8);
      }
#pragma unroll
      for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int part = 0; part < 2; ++part) {
          const __nv_bfloat16 *qr = (part ? qo : qh) + (16 * mt + gr) * RS + k0 + gc;
          const uint32_t a0 = *(const uint32_t *)qr, a1 = *(const uint32_t *)(qr + 8 * RS);
          const uint32_t a2 = *(const uint32_t *)(qr + 8), a3 = *(const uint32_t *)(qr + 8 * RS + 8);
#pragma unroll
          for (int nt = 0; nt < 2; ++nt) sel_mma_bf16(acc[mt][nt], a0, a1, a2, a3, b[nt][0], b[nt][1]);
        }
    }
    __syncthreads();  // keys consumed: lt reuses their space
    if (tid == 0) trace_mark(1);  // logits computed
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int ql = 16 * mt + gr + (e >> 1) * 8, kk = 16 * warp + 8 * nt + gc + (e & 1);
          const float l = acc[mt][nt][e] * scale;
          lt[ql * SEL_LTS + kk] = kk < nk ? l : -INFINITY;
          if (kk < nk && ql < nq) ws.logit[(qg0 + ql) * c + t0 + kk] = l;
        }
  } else {
    // fp32 keys: FFMA micro-tiles.  Both operands transposed, d-major: the
    // thread of micro-tile (queries 4qg.., keys 4kg..) reads one float4 of
    // each per d
    float *qT = (float *)sel_smem;   // [dh][SEL_QT]
    float *kT = qT + dh * SEL_QT;    // [dh][SEL_KC]
    lt = kT;
    last = (int *)qT;
    // the pool's stale keys: no kernel of the pass writes them, so they are
    // read before the wait on the predecessor; a thread issues all its loads
    // (page lookups, then rows) before it uses the first
    constexpr int EPV = 16 / (int)sizeof(T);  // elements per 16-byte load
    constexpr int KLD = SEL_KC * (SEL_DH_MAX / EPV) / SEL_THREADS;
    const T *kc = (const T *)v.pages;
    const int L = dh / EPV;
    uint4 kx[KLD];
#pragma unroll
    for (int u = 0; u < KLD; ++u) {
      const int i = tid + u * SEL_THREADS, kk = i % SEL_KC, sub = i / SEL_KC;
      kx[u] = make_uint4(0u, 0u, 0u, 0u);
      if (kk < nk && sub < L)
        kx[u] = *(const uint4 *)(kc + v.offset(layer, 0, g, s_end + t0 + kk) + sub * EPV);
    }
#pragma unroll
    for (int u = 0; u < KLD; ++u) {
      const int i = tid + u * SEL_THREADS, kk = i % SEL_KC, sub = i / SEL_KC;
      if (sub < L) {
        const float *f = (const float *)&kx[u];
#pragma unroll
        for (int e = 0; e < EPV; ++e) kT[(sub * EPV + e) * SEL_KC + kk] = f[e];  // lanes: consecutive keys
      }
    }
    pdl_wait();  // the queries come from the RoPE kernel just before
    ts.waited();
    constexpr int QLD = SEL_QT * (SEL_DH_MAX / 4) / SEL_THREADS;
    const int D4 = dh / 4;
    float4 qx[QLD];
#pragma unroll
    for (int u = 0; u < QLD; ++u) {
      const int i = tid + u * SEL_THREADS, ql = i % SEL_QT, d4 = i / SEL_QT;
      qx[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (ql < nq && d4 < D4) {
        const int qq = q0 + ql, r = qq / hpg, hh = g * hpg + qq % hpg;
        qx[u] = *(const float4 *)(q + ((size_t)r * H + hh) * dh + 4 * d4);
      }
    }
#pragma unroll
    for (int u = 0; u < QLD; ++u) {
      const int i = tid + u * SEL_THREADS, ql = i % SEL_QT, d4 = i / SEL_QT;
      if (d4 < D4) {
        float *dst = qT + 4 * d4 * SEL_QT + ql;  // lanes: consecutive queries
        dst[0] = qx[u].x;
        dst[SEL_QT] = qx[u].y;
        dst[2 * SEL_QT] = qx[u].z;
        dst[3 * SEL_QT] = qx[u].w;
      }
    }
    __syncthreads();
    if (tid == 0) trace_mark(0);  // keys and queries staged
    const int kg = tid % SEL_KG, qg = tid / SEL_KG;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
#pragma unroll 4
    for (int d = 0; d < dh; ++d) {
      const float4 a = *(const float4 *)(qT + d * SEL_QT + 4 * qg);
      const float4 b = *(const float4 *)(kT + d * SEL_KC + 4 * kg);
      const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();  // keys consumed: lt reuses their space
    if (tid == 0) trace_mark(1);  // logits computed
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int ql = 4 * qg + i;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int kk = 4 * kg + j;
        const float l = acc[i][j] * scale;
        lt[ql * SEL_LTS + kk] = kk < nk ? l : -INFINITY;
        if (kk < nk && ql < nq) ws.logit[(qg0 + ql) * c + t0 + kk] = l;
      }
    }
  }
  __syncthreads();
  // chunk statistics: 4 threads per query, keys o, o + 4, ... (the row
  // stride SEL_LTS = 4 mod 32 puts a warp's 8 queries x 4 lanes on 32 banks)
  const int ql = tid >> 2, o = tid & 3;
  {
    const float *row = lt + ql * SEL_LTS;
    float mx = -INFINITY;
#pragma unroll
    for (int j = 0; j < SEL_KC / 4; ++j) mx = fmaxf(mx, row[o + 4 * j]);
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    float z = 0.f;  // key 0 is valid: mx is finite
#pragma unroll
    for (int j = 0; j < SEL_KC / 4; ++j) z += expf(row[o + 4 * j] - mx);
    z += __shfl_xor_sync(0xffffffffu, z, 2);
    z += __shfl_xor_sync(0xffffffffu, z, 1);
    if (o == 0 && ql < nq) ws.ml[(qg0 + ql) * nch + chunk] = make_float2(mx, z);
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) trace_mark(2);  // chunk statistics stored
  int *cnt = ws.cnt + (size_t)g * gridDim.z + qt;
  if (tid == 0) *last = atomicAdd(cnt, 1) == nch - 1;
  __syncthreads();
  if (tid == 0) trace_mark(3);  // arrival counted
  if (!*last) return;
  if (tid == 0) *cnt = 0;  // ready for the next layer's launch
  __threadfence();
  // fold: 4 threads per query, each over chunks o, o + 4, ... (SEL_FOLD
  // loads in flight), then the quad
  float mx = -INFINITY, z = 0.f;
  if (ql < nq) {
    const float2 *row = ws.ml + (qg0 + ql) * nch;
    for (int base = o; base < nch; base += 4 * SEL_FOLD) {
      float2 x[SEL_FOLD];
#pragma unroll
      for (int j = 0; j < SEL_FOLD; ++j) {
        const int ch = base + 4 * j;
        x[j] = ch < nch ? __ldcg(row + ch) : make_float2(-INFINITY, 0.f);
      }
#pragma unroll
      for (int j = 0; j < SEL_FOLD; ++j) lse_merge(mx, z, x[j].x, x[j].y);
    }
  }
#pragma unroll
  for (int off = 2; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, mx, off);
    const float z2 = __shfl_xor_sync(0xffffffffu, z, off);
    lse_merge(mx, z, m2, z2);
  }
  if (o == 0 && ql < nq) ws.mz[qg0 + ql] = make_float2(mx, 1.0f / z);
  if (tid == 0) trace_mark(4);  // fold done (last CTA of the group)
}

// score[j] += sum over the S*H queries of exp(logit - max) / sum, in a fixed
// order: a CTA takes ACC_KEYS keys; its ACC_SLICES thread slices sum
// interleaved sets of the queries (coalesced along the keys), then one
// thread per key adds the slice sums in slice order.
constexpr int ACC_KEYS = 16, ACC_SLICES = 32;
__global__ void __launch_bounds__(ACC_KEYS * ACC_SLICES)
    k_attn_select_accum(const float *logit, const float2 *mz, int NQ, int c, int s_end,
                        float *score) {
  TraceScope ts(TK_SELECT_ACC);
  pdl_trigger();
  __shared__ float part[ACC_SLICES][ACC_KEYS];
  const int kk = threadIdx.x % ACC_KEYS, sl = threadIdx.x / ACC_KEYS;
  const int t = blockIdx.x * ACC_KEYS + kk;
  pdl_wait();  // logits and softmax statistics of the kernel before
  float s = 0.f;
  if (t < c) {
#pragma unroll 8
    for (int qg = sl; qg < NQ; qg += ACC_SLICES) {
      const float2 st = mz[qg];
      s += expf(logit[(size_t)qg * c + t] - st.x) * st.y;
    }
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

void launch_first_delim(const int32_t *tokens, int n, int s_end, int delim, int *bound,
                        cudaStream_t s) {
  int c = n - s_end;
  if (c <= 0) return;
  k_first_delim<<<grid_for(c, 256), 256, 0, s>>>(tokens, n, s_end, delim, bound);
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
                        int32_t *count, cudaStream_t s, const SimpleKeys &gen,
                        const int *flag_in, int32_t *flag_out) {
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
  k_topk<<<1, TOPK_THREADS, smem, s>>>(keys, c, s_end, K, nonzero_only, out, count, gen,
                                       flag_in, flag_out);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

namespace {
struct SelLayout {
  size_t logit, ml, mz, cnt, total;  // byte offsets into the workspace
};
SelLayout sel_layout(int S, const Dims &dm, int c) {
  auto al = [](size_t x) { return (x + 255) / 256 * 256; };
  const size_t NQ = (size_t)S * dm.H, nqt = ((size_t)S * (dm.H / dm.G) + SEL_QT - 1) / SEL_QT;
  SelLayout o;
  o.logit = 0;
  o.ml = o.logit + al(NQ * c * sizeof(float));
  o.mz = o.ml + al(NQ * sel_chunks(c) * sizeof(float2));
  o.cnt = o.mz + al(NQ * sizeof(float2));
  o.total = o.cnt + al((size_t)dm.G * nqt * sizeof(int));
  return o;
}
}  // namespace

size_t attn_select_ws_bytes(int S, const Dims &dm, int n_pool) {
  return n_pool > 0 && S > 0 ? sel_layout(S, dm, n_pool).total : 0;
}

void launch_attn_select_scores(const float *q, int S, const Dims &dm, int layer, KVView v,
                               int s_end, int n, void *ws_base, bool first_layer,
                               float *scores, cudaStream_t s) {
  const int c = n - s_end;
  if (c <= 0 || S <= 0) return;
  const float scale = (float)(1.0 / sqrt((double)dm.dh));
  const SelLayout o = sel_layout(S, dm, c);
  char *b = (char *)ws_base;
  SelWs ws{(float *)(b + o.logit), (float2 *)(b + o.ml), (float2 *)(b + o.mz), (int *)(b + o.cnt)};
  const int nqt = (S * (dm.H / dm.G) + SEL_QT - 1) / SEL_QT;
  // arrival counts start at zero; each launch's last CTAs leave them at zero
  if (first_layer) cudaMemsetAsync(ws.cnt, 0, (size_t)dm.G * nqt * sizeof(int), s);
  const dim3 grid(sel_chunks(c), dm.G, nqt);
  // bf16: q_hi, q_lo and keys as bf16 rows of dh + 8; fp32: q and keys as
  // fp32 columns of dh.  The logits tile reuses the keys' space.
  const bool bf16 = dm.dtype == KVR_DTYPE_BF16;
  const size_t q_b = bf16 ? (size_t)2 * SEL_QT * (dm.dh + 8) * 2 : (size_t)SEL_QT * dm.dh * 4;
  const size_t k_b = bf16 ? (size_t)SEL_KC * (dm.dh + 8) * 2 : (size_t)SEL_KC * dm.dh * 4;
  const size_t lt_b = (size_t)SEL_QT * SEL_LTS * sizeof(float);
  const size_t smem = q_b + (k_b > lt_b ? k_b : lt_b);  // 34 KB (bf16), 48 KB (fp32) at dh 128
  auto kern = bf16 ? k_attn_select_logits<__nv_bfloat16> : k_attn_select_logits<float>;
  // fp32 at dh 128, plus the trace build's static shared memory, passes 48 KB
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  launch_pdl(kern, grid, SEL_THREADS, smem, s, q, S, dm.H, dm.G, dm.dh, layer, v, s_end, c, scale,
             ws);
  launch_pdl(k_attn_select_accum, (c + ACC_KEYS - 1) / ACC_KEYS, ACC_KEYS * ACC_SLICES, 0, s,
             (const float *)ws.logit, (const float2 *)ws.mz, S * dm.H, c, s_end, scores);
}

void launch_kv_deviation(const float *qkv, const float2 *rope, const int32_t *pos, int M,
                         const Dims &dm, KVView v, float *scores, cudaStream_t s) {
  if (M <= 0) return;
  if (dm.dtype == KVR_DTYPE_BF16)
    k_kv_deviation<__nv_bfloat16><<<M, 256, 0, s>>>(qkv, rope, pos, dm.H, dm.G, dm.dh, v, scores);
  else
    k_kv_deviation<float><<<M, 256, 0, s>>>(qkv, rope, pos, dm.H, dm.G, dm.dh, v, scores);
}

KVR_TRACE_ATTACH(trace_attach_select)

}  // namespace kvr
