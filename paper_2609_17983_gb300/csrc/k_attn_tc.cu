// k_attn_tc.cu -- scattered-query causal GQA attention on tensor cores, bf16
// cache, split over keys (flash-decoding style) for the few-row repair pass
// and unsplit for prefill-size passes.
//
// A CTA owns one query block -- consecutive rows of one document, times the
// grp = H/G query heads that share KV head g, at most 192 query vectors, one
// warp per 16 -- and
// a contiguous range of 64-key chunks (one KV page each).  It streams the K
// and V pages of its range through double-buffered cp.async into XOR-swizzled
// shared memory, computes S = Q K^T and O += P V with mma.sync m16n8k16 (bf16
// in, fp32 accumulate), masks key j > position of the query row, and keeps the
// softmax online (running max in the log2 domain).  With several key splits
// each CTA writes its unnormalised O and (max, sum) and a combine kernel
// merges the splits in split order (deterministic).
//
// Rows of the pass were written into the cache at this layer before the
// launch, so every row sees the fresh K/V of the others and stale K/V
// elsewhere (operator R, Sec. 3).
#include <math.h>

#include <algorithm>
#include <cmath>

#include <type_traits>

#include "kvr_internal.cuh"

namespace kvr {
namespace {

constexpr int CHUNK = KVR_PAGE;  // keys per chunk = one page
constexpr int MAXW = 12;         // warps per CTA, 16 query vectors each
constexpr int MAXQ = MAXW * 16;  // query vectors per CTA

struct AttnTcParams {
  const __nv_bfloat16 *q;  // [M][H*dh] post-RoPE
  float qk_scale;          // log2(e) / sqrt(dh): scores into the log2 domain
  int H, G, grp;
  const int32_t *pos;
  const int4 *blocks;  // (row0, nrows, kmax, doc)
  int layer;
  KVView single;
  const KVView *views;
  int n_splits;
  float *ws_o;   // [n_splits][n_blocks][MAXQ][dh]
  float2 *ws_ml; // [n_splits][n_blocks][MAXQ]
  int n_blocks;
  __nv_bfloat16 *out;  // [M][H*dh]
  int cq;              // query slots per (block, head) the combine visits: the largest block's
  const char *pf;      // weights of the next GEMM, warmed into L2 by the combine (HBM is idle)
  long long pf_bytes;
};

__device__ __forceinline__ uint32_t su32(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                          uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma16816(float *d, uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *(uint32_t *)&v;
}

// byte offset of 16-byte chunk c of row r in a swizzled [rows][DH] bf16 tile
template <int DH>
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return (uint32_t)(r * DH * 2 + ((c ^ (r & 7)) << 4));
}

template <int DH>
__global__ void __launch_bounds__(MAXW * 32, 1) k_attn_tc(const AttnTcParams p) {
  constexpr int NCH = DH / 8;        // 16-byte chunks per row
  constexpr int KT = DH / 16;        // k-steps of QK^T
  constexpr int OT = DH / 8;         // n-tiles of O
  constexpr int TILE = CHUNK * DH * 2;
  extern __shared__ __align__(128) uint8_t sm[];
  uint8_t *sQ = sm;                            // MAXQ x DH
  uint8_t *sK = sm + MAXQ * DH * 2;            // 2 x CHUNK x DH
  uint8_t *sV = sK + 2 * TILE;                 // 2 x CHUNK x DH
  __shared__ int spos[MAXQ];

  TraceScope ts(TK_ATTN);
  pdl_trigger();
  // The block table, positions and page table are written before the pass;
  // the cache pages are final except for the pass's own rows, which the RoPE
  // kernel writes.  So everything up to the wait may read them, and the key
  // range of this CTA is pulled into L2 meanwhile (the RoPE writes land in
  // the same L2 lines).
  const int split = blockIdx.x, g = blockIdx.y, blk = blockIdx.z;
  const int4 bd = p.blocks[blk];
  const int row0 = bd.x, nrows = bd.y, kmax = bd.z;
  const KVView kv = p.views ? p.views[bd.w] : p.single;
  const int mq = nrows * p.grp;
  const int n_chunks = kmax / CHUNK + 1;
  const int cps = (n_chunks + p.n_splits - 1) / p.n_splits;
  const int c0 = split * cps, c1 = min(n_chunks, c0 + cps);
  if (c0 >= c1) return;  // empty split: the combine skips it
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nthr = blockDim.x, nq = blockDim.x >> 1;  // query vectors of this launch
  const __nv_bfloat16 *cache = (const __nv_bfloat16 *)kv.pages;
  if (tid < 2 * (c1 - c0)) {
    const __nv_bfloat16 *pg = cache + kv.offset(p.layer, tid & 1, g, (c0 + (tid >> 1)) * CHUNK);
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(pg), "r"(TILE) : "memory");
  }
  for (int v = tid; v < nq; v += nthr) spos[v] = v < mq ? p.pos[row0 + v / p.grp] : -1;
  pdl_wait();
  ts.waited();

  auto load_chunk = [&](int c, int buf) {
    const __nv_bfloat16 *kp = cache + kv.offset(p.layer, 0, g, c * CHUNK);
    const __nv_bfloat16 *vp = cache + kv.offset(p.layer, 1, g, c * CHUNK);
    uint32_t kb = su32(sK + buf * TILE), vb = su32(sV + buf * TILE);
    for (int e = tid; e < CHUNK * NCH; e += nthr) {
      int r = e / NCH, ch = e % NCH;
      cp_async16(kb + swz<DH>(r, ch), kp + r * DH + ch * 8);
      cp_async16(vb + swz<DH>(r, ch), vp + r * DH + ch * 8);
    }
    cp_commit();
  };

  // Q block (bf16, already scaled) straight into swizzled shared memory,
  // committed with the first chunk
  {
    const uint32_t qb = su32(sQ);
    for (int e = tid; e < nq * NCH; e += nthr) {
      int v = e / NCH, ch = e % NCH;
      if (v < mq) {
        int r = row0 + v / p.grp, hh = g * p.grp + v % p.grp;
        cp_async16(qb + swz<DH>(v, ch), p.q + ((size_t)r * p.H + hh) * DH + ch * 8);
      } else {
        *(uint4 *)(sQ + swz<DH>(v, ch)) = make_uint4(0, 0, 0, 0);
      }
    }
  }
  load_chunk(c0, 0);

  const bool active = warp * 16 < mq;
  const int v0 = warp * 16 + (lane >> 2), v1 = v0 + 8;
  float o[OT][4];
#pragma unroll
  for (int i = 0; i < OT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  __syncthreads();
  const int p0 = spos[v0], p1 = spos[v1];

  for (int c = c0; c < c1; ++c) {
    const int buf = (c - c0) & 1;
    if (c + 1 < c1) {
      load_chunk(c + 1, buf ^ 1);
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();
    if (active) {
      const uint32_t qb = su32(sQ), kb = su32(sK + buf * TILE), vb = su32(sV + buf * TILE);
      float s[8][4];
#pragma unroll
      for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < KT; ++ks) {
        uint32_t a0, a1, a2, a3;
        ldsm_x4(qb + swz<DH>(warp * 16 + (lane & 15), 2 * ks + (lane >> 4)), a0, a1, a2, a3);
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4(kb + swz<DH>(16 * np + (lane & 7) + ((lane >> 4) << 3),
                               2 * ks + ((lane >> 3) & 1)),
                  b0, b1, b2, b3);
          mma16816(s[2 * np], a0, a1, a2, a3, b0, b1);
          mma16816(s[2 * np + 1], a0, a1, a2, a3, b2, b3);
        }
      }
      // causal mask on original positions, online softmax (log2 domain)
      // against integer reference maxima, so that bf16(P) is a power of two
      // times the rounding of 2^(x - E) for any integer E
      const int kbase = c * CHUNK + 2 * (lane & 3);
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        int j = kbase + 8 * nt;
#pragma unroll
        for (int k = 0; k < 4; ++k) s[nt][k] *= p.qk_scale;
        if (j > p0) s[nt][0] = -INFINITY;
        if (j + 1 > p0) s[nt][1] = -INFINITY;
        if (j > p1) s[nt][2] = -INFINITY;
        if (j + 1 > p1) s[nt][3] = -INFINITY;
        mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]));
        mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]));
      }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float mn0 = fmaxf(m0, ceilf(mx0)), mn1 = fmaxf(m1, ceilf(mx1));
      const float b0s = mn0 == -INFINITY ? 0.f : mn0, b1s = mn1 == -INFINITY ? 0.f : mn1;
      const float cr0 = exp2f(m0 - b0s), cr1 = exp2f(m1 - b1s);
      m0 = mn0;
      m1 = mn1;
      float rs0 = 0.f, rs1 = 0.f;
      uint32_t pa[8][2];
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        float e0 = exp2f(s[nt][0] - b0s), e1 = exp2f(s[nt][1] - b0s);
        float e2 = exp2f(s[nt][2] - b1s), e3 = exp2f(s[nt][3] - b1s);
        rs0 += e0 + e1;
        rs1 += e2 + e3;
        pa[nt][0] = pack_bf16(e0, e1);
        pa[nt][1] = pack_bf16(e2, e3);
      }
      l0 = l0 * cr0 + rs0;
      l1 = l1 * cr1 + rs1;
#pragma unroll
      for (int i = 0; i < OT; ++i) {
        o[i][0] *= cr0;
        o[i][1] *= cr0;
        o[i][2] *= cr1;
        o[i][3] *= cr1;
      }
      // O += P V
#pragma unroll
      for (int ks = 0; ks < CHUNK / 16; ++ks) {
        const uint32_t a0 = pa[2 * ks][0], a1 = pa[2 * ks][1], a2 = pa[2 * ks + 1][0],
                       a3 = pa[2 * ks + 1][1];
#pragma unroll
        for (int np = 0; np < OT / 2; ++np) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(vb + swz<DH>(16 * ks + (lane & 7) + (((lane >> 3) & 1) << 3),
                                 2 * np + (lane >> 4)),
                    b0, b1, b2, b3);
          mma16816(o[2 * np], a0, a1, a2, a3, b0, b1);
          mma16816(o[2 * np + 1], a0, a1, a2, a3, b2, b3);
        }
      }
    }
    __syncthreads();  // buffer buf is refilled by the next iteration's prefetch
  }
  if (threadIdx.x == 0) trace_mark(0);
  if (!active) return;
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const int dcol = 2 * (lane & 3);
  if (p.n_splits == 1) {
    const float i0 = l0 > 0.f ? 1.f / l0 : 0.f, i1 = l1 > 0.f ? 1.f / l1 : 0.f;
#pragma unroll
    for (int nt = 0; nt < OT; ++nt) {
      int d = 8 * nt + dcol;
      if (v0 < mq) {
        int r = row0 + v0 / p.grp, hh = g * p.grp + v0 % p.grp;
        *(uint32_t *)(p.out + ((size_t)r * p.H + hh) * DH + d) =
            pack_bf16(o[nt][0] * i0, o[nt][1] * i0);
      }
      if (v1 < mq) {
        int r = row0 + v1 / p.grp, hh = g * p.grp + v1 % p.grp;
        *(uint32_t *)(p.out + ((size_t)r * p.H + hh) * DH + d) =
            pack_bf16(o[nt][2] * i1, o[nt][3] * i1);
      }
    }
  } else {
    // ws index: split-major, then (block, kv head) pair, then query vector
    const size_t bs = ((size_t)split * p.n_blocks + blk) * p.G + g;
    float *wo = p.ws_o + bs * MAXQ * DH;  // per (split, block, head): MAXQ x DH
#pragma unroll
    for (int nt = 0; nt < OT; ++nt) {
      int d = 8 * nt + dcol;
      *(float2 *)(wo + (size_t)v0 * DH + d) = make_float2(o[nt][0], o[nt][1]);
      *(float2 *)(wo + (size_t)v1 * DH + d) = make_float2(o[nt][2], o[nt][3]);
    }
    if ((lane & 3) == 0) {
      p.ws_ml[bs * MAXQ + v0] = make_float2(m0, l0);
      p.ws_ml[bs * MAXQ + v1] = make_float2(m1, l1);
    }
  }
}

// Merge the key splits of every (block, kv head, query vector), in split
// order.  Two warps per query vector, each owning half of head_dim: lane s
// reads split s's (max, sum), the weights are reduced across the warp, and
// the partial outputs of up to NB splits load in one round trip with few
// registers (so the next GEMM's CTAs can be resident, and stream their first
// weight tiles, while this kernel runs).
template <int DH>
__global__ void __launch_bounds__(256) k_attn_combine(const AttnTcParams p) {
  TraceScope ts(TK_COMBINE);
  pdl_trigger();
  if (p.pf_bytes > 0) {
    // this CTA's slice of the next GEMM's weights, in pieces of PF_PIECE bytes
    constexpr long long PF_PIECE = 32 << 10;
    const long long slice = (p.pf_bytes / gridDim.x + 15) & ~15ll;
    const long long b0 = (long long)blockIdx.x * slice;
    const long long b1 = min(p.pf_bytes, b0 + slice);
    for (long long o = b0 + (long long)threadIdx.x * PF_PIECE; o < b1; o += 256 * PF_PIECE) {
      const long long n = min(PF_PIECE, b1 - o) & ~15ll;
      if (n > 0)
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p.pf + o), "r"((int)n)
                     : "memory");
    }
  }
  pdl_wait();
  ts.waited();
  const int gw = (blockIdx.x * 8) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  const int half = gw & 1, wv = gw >> 1;
  const int total = p.n_blocks * p.G * p.cq;
  if (wv >= total) return;
  const int v = wv % p.cq, bg = wv / p.cq;
  const int g = bg % p.G, blk = bg / p.G;
  const int4 bd = p.blocks[blk];
  const int mq = bd.y * p.grp;
  if (v >= mq) return;
  const int n_chunks = bd.z / CHUNK + 1;
  const int cps = (n_chunks + p.n_splits - 1) / p.n_splits;
  const int ns = (n_chunks + cps - 1) / cps;  // non-empty splits
  const size_t stride = (size_t)p.n_blocks * p.G;  // between splits, in (block, head) units
  const size_t base = (size_t)blk * p.G + g;
  constexpr int VPL = DH / 64;  // floats per lane
  constexpr int NB = 12;        // splits whose partial outputs load in the first round trip
  using VecT = typename std::conditional<VPL == 2, float2, float>::type;
  const VecT *src = (const VecT *)(p.ws_o + (base * MAXQ + v) * DH + half * (DH / 2)) + lane;
  const size_t sstride = stride * MAXQ * DH / VPL;  // in vectors
  VecT x[NB];
#pragma unroll
  for (int j = 0; j < NB; ++j)
    if (j < ns) x[j] = __ldcg(src + j * sstride);
  // (max, sum) of up to 64 splits, two per lane
  float2 ml0 = lane < ns ? p.ws_ml[(base + lane * stride) * MAXQ + v] : make_float2(-INFINITY, 0.f);
  float2 ml1 = lane + 32 < ns ? p.ws_ml[(base + (lane + 32) * stride) * MAXQ + v]
                              : make_float2(-INFINITY, 0.f);
  float mx = fmaxf(ml0.y > 0.f ? ml0.x : -INFINITY, ml1.y > 0.f ? ml1.x : -INFINITY);
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  const float w0 = ml0.y > 0.f ? exp2f(ml0.x - mx) : 0.f;
  const float w1 = ml1.y > 0.f ? exp2f(ml1.x - mx) : 0.f;
  float l = w0 * ml0.y + w1 * ml1.y;
  for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
  float acc[VPL];
#pragma unroll
  for (int i = 0; i < VPL; ++i) acc[i] = 0.f;
  // in split order, as the partials of split j carry weight w_j
#pragma unroll
  for (int j = 0; j < NB; ++j) {
    const float w = __shfl_sync(0xffffffffu, w0, j & 31);
    if (j < ns) {
      const float *xv = (const float *)&x[j];
#pragma unroll
      for (int i = 0; i < VPL; ++i) acc[i] += w * xv[i];
    }
  }
  for (int sj = NB; sj < ns; ++sj) {
    const float w = __shfl_sync(0xffffffffu, sj < 32 ? w0 : w1, sj & 31);
    const VecT y = __ldcg(src + sj * sstride);
    const float *yv = (const float *)&y;
#pragma unroll
    for (int i = 0; i < VPL; ++i) acc[i] += w * yv[i];
  }
  const float inv = l > 0.f ? 1.f / l : 0.f;
  const int r = bd.x + v / p.grp, hh = g * p.grp + v % p.grp;
  __nv_bfloat16 *dst = p.out + ((size_t)r * p.H + hh) * DH + half * (DH / 2) + lane * VPL;
  if constexpr (VPL == 2)
    *(uint32_t *)dst = pack_bf16(acc[0] * inv, acc[1] * inv);
  else
    *dst = __float2bfloat16_rn(acc[0] * inv);
}

template <int DH>
const char *run(const AttnTcParams &p, int max_mq, cudaStream_t s) {
  constexpr int smem = MAXQ * DH * 2 + 4 * CHUNK * DH * 2;
  const int warps = (max_mq + 15) / 16;
  static bool set = false;
  if (!set) {
    cudaError_t e = cudaFuncSetAttribute(k_attn_tc<DH>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cudaGetErrorString(e);
    set = true;
  }
  dim3 grid(p.n_splits, p.G, p.n_blocks);
  launch_pdl(k_attn_tc<DH>, grid, warps * 32, smem, s, p);
  if (p.n_splits > 1) {
    int warps = 2 * p.n_blocks * p.G * p.cq;
    launch_pdl(k_attn_combine<DH>, (warps + 7) / 8, 256, 0, s, p);
  }
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

template <int DH>
const char *run_combine(const AttnTcParams &p, cudaStream_t s) {
  const int warps = 2 * p.n_blocks * p.G * p.cq;
  launch_pdl(k_attn_combine<DH>, (warps + 7) / 8, 256, 0, s, p);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

}  // namespace

const char *launch_attention_combine(const int4 *blocks, int n_blocks, int max_rows_per_block,
                                     int n_splits, const Dims &dm, float *ws_o, float2 *ws_ml,
                                     void *out, cudaStream_t s, const void *prefetch,
                                     long long prefetch_bytes) {
  if (n_blocks <= 0 || n_splits <= 1) return nullptr;
  AttnTcParams p{};
  p.pf = (const char *)prefetch;
  p.pf_bytes = prefetch && ((uintptr_t)prefetch & 15) == 0 ? prefetch_bytes : 0;
  p.cq = std::min(MAXQ, max_rows_per_block * (dm.H / dm.G));
  p.H = dm.H;
  p.G = dm.G;
  p.grp = dm.H / dm.G;
  p.blocks = blocks;
  p.n_splits = n_splits;
  p.ws_o = ws_o;
  p.ws_ml = ws_ml;
  p.n_blocks = n_blocks;
  p.out = (__nv_bfloat16 *)out;
  if (dm.dh == 128) return run_combine<128>(p, s);
  if (dm.dh == 64) return run_combine<64>(p, s);
  return "head_dim not supported";
}

int attn_tc_rows_per_block(int grp) { return MAXQ / grp; }

size_t attn_tc_ws_floats(int n_splits, int n_blocks, int G, int dh) {
  return (size_t)n_splits * n_blocks * G * MAXQ * dh;
}

const char *launch_attention_tc(const void *q, const int32_t *pos, const int4 *blocks,
                                int n_blocks, int max_rows_per_block, int n_splits, const Dims &dm,
                                int layer, const KVView *views, KVView single, float *ws_o,
                                float2 *ws_ml, void *out, cudaStream_t s) {
  if (n_blocks <= 0) return nullptr;
  AttnTcParams p{};
  p.q = (const __nv_bfloat16 *)q;
  p.qk_scale = (float)(1.4426950408889634 / std::sqrt((double)dm.dh));
  p.H = dm.H;
  p.G = dm.G;
  p.grp = dm.H / dm.G;
  p.pos = pos;
  p.blocks = blocks;
  p.layer = layer;
  p.single = single;
  p.views = views;
  p.n_splits = n_splits;
  p.ws_o = ws_o;
  p.ws_ml = ws_ml;
  p.n_blocks = n_blocks;
  p.out = (__nv_bfloat16 *)out;
  const int max_mq = max_rows_per_block * p.grp;
  p.cq = max_mq;
  if (dm.dh == 128) return run<128>(p, max_mq, s);
  if (dm.dh == 64) return run<64>(p, max_mq, s);
  return "head_dim not supported";
}

KVR_TRACE_ATTACH(trace_attach_attn)

}  // namespace kvr
