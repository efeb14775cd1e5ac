// k_attn_tc5.cu -- scattered-query causal GQA attention of one document's
// rows on the tcgen05 tensor cores (sm_103a), bf16 cache, head_dim 64 or 128.
//
// A CTA owns one query block -- up to 128 query vectors (rows of the pass times
// the grp query heads of KV head g, all of one document), the M = 128 rows of
// the MMA -- and a contiguous range of 64-key chunks (one KV page each).  A
// pass over several documents gives each its own page table and TMA view.  Per chunk:
//   S = Q K^T      tcgen05.mma, M 128 x N 64 x K head_dim, into TMEM (two
//                  S buffers, so S of chunk i+1 is computed while the softmax
//                  works on chunk i);
//   softmax        sixteen warps, four per TMEM lane quarter: one query
//                  vector per four threads, each thread a quarter of the
//                  chunk's keys and of O's columns (four warps per SM
//                  sub-partition hide each other's latency), the row maximum
//                  exchanged through shared memory; S read once from
//                  TMEM: causal mask key <= position, scores scaled by
//                  log2(e)/sqrt(dh) into the log2 domain, exponentials
//                  against an integer reference maximum that is raised -- and
//                  the accumulator rescaled in TMEM by a power of two -- only
//                  when the running maximum exceeds it by more than 8 (so
//                  P <= 256); with an integer reference, bf16(P) is a power
//                  of two times the rounding of 2^(x - E) for any integer E,
//                  whichever chunk set it; P in bf16 written with
//                  tcgen05.st to one of two tensor-memory buffers as the next
//                  MMA's A operand, so the softmax of chunk i overlaps
//                  O += P V of chunk i-1;
//   O += P V       tcgen05.mma, M 128 x N head_dim x K 64, V read MN-major
//                  straight from the page layout [key][head_dim].
// Both MMAs take A (Q, then P) from tensor memory and only B (K, then V) from
// shared memory, so a chunk's shared-memory traffic is its K and V tiles, each
// written once by TMA and read once by an MMA.  K and V tiles arrive by TMA
// (128-byte swizzle, KV_STAGES stages deep, so a chunk's load is issued long
// before its MMA); the softmax warps write Q into tensor memory once.
// With several key splits the CTA writes its unnormalised O and (max, sum)
// for the combine kernel, else the normalised output.
//
// Rows of the pass were written into the cache at this layer before the
// launch (operator R, Sec. 3); keys are read only after the wait on that
// kernel, and only L2 prefetches are issued before it.
//
// Warp roles (576 threads): warp 0 TMA (one lane), warp 1 TMEM allocation and
// MMA issue (one lane), warps 2-17 softmax and epilogue.  Every wait is
// bounded; a wait that runs out sets the device error flag, the roles stop
// issuing, drain what is in flight, free TMEM and return.
#include <math.h>

#include "kvr_internal.cuh"
#include "tc_ptx.cuh"

namespace kvr {
namespace {
using namespace ptx;

constexpr int QV = 128;          // query vectors per CTA (UMMA M)
constexpr int CH = KVR_PAGE;     // keys per chunk
constexpr int SMW = 4;           // softmax warps per TMEM lane quarter
constexpr int NT5 = 64 + 128 * SMW;  // threads per CTA
constexpr int WS_MAXQ = 192;     // query slots per (split, block, head) of the split workspace
// Tensor-memory columns: S buffers at 0 and 64, O (head_dim columns) at 128,
// Q (head_dim / 2 columns of bf16 pairs) at T_Q, P buffers (32 columns each) at T_P.
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t T_Q = 256, T_P = 320;
// Holding all of TMEM cannot stall on another grid: the other kernel that
// allocates TMEM (the GEMM) cannot share an SM with this one (their register
// files together exceed the SM's), and dependents launch only after every CTA
// here holds its columns.
constexpr int SOFTMAX_THREADS = 128 * SMW;
constexpr float RESCALE_LOG2 = 8.f;  // headroom of the reference maximum (P <= 2^8)
constexpr int KV_STAGES = 4;

struct Attn5Params {
  const __nv_bfloat16 *q;  // [M][H * dh] post-RoPE
  float qk_scale;          // log2(e) / sqrt(dh): scores into the log2 domain
  const int32_t *pos;      // [M] ascending (one document)
  const int4 *blocks;      // (row0, nrows, kmax, doc)
  const __nv_bfloat16 *pages;  // the cache's page pool (one document)
  const int32_t *table;        // logical page -> physical page (one document)
  // several documents: their views and the TMA views of their page pools
  // (device memory, 64-byte aligned), indexed by the block's document
  const KVView *views;
  const CUtensorMap *tmaps;
  int H, G, grp, layer, L;
  int n_splits, n_blocks;
  float *ws_o;    // [n_splits][n_blocks][G][WS_MAXQ][dh]
  float2 *ws_ml;  // [n_splits][n_blocks][G][WS_MAXQ]
  __nv_bfloat16 *out;  // [M][H * dh]
  int *dev_flag;
};

// A from tensor memory: row m of A in TMEM lane m, two bf16 of K per 32-bit
// column (K-major), a_tmem the column of its first K element; B a shared-memory
// descriptor.
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}

// 8 consecutive 32-bit TMEM columns of the warp's 32 lanes, one lane per
// thread, without the wait (tmem_wait_st before the data is consumed).
__device__ __forceinline__ void tmem_st8_nowait(uint32_t taddr, const uint32_t *r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *(uint32_t *)&v;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int DH>
__global__ void __launch_bounds__(NT5, 1)
    k_attn_tc5(const __grid_constant__ CUtensorMap tm_kv, const Attn5Params p) {
  constexpr int HALVES = DH / 64;           // 128-byte column blocks of a row
  constexpr uint32_t TBYTES = CH * 128 * HALVES;  // one K (or V) tile
  constexpr uint32_t KVBYTES = 2 * TBYTES;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t kv_full[KV_STAGES], kv_empty[KV_STAGES], s_full[2], s_free[2],
      p_full[2], o_done[2], q_full, drain_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_f;
  __shared__ int spos[QV];
  __shared__ int sprow[2 * 64];  // pool rows of the CTA's K and V pages (at most 64 chunks)
  __shared__ float sx[2][SMW][QV];  // per chunk parity and key part: row maxima
  __shared__ float ssum[SMW][QV];   // per key part: sums of exponentials

  TraceScope ts(TK_ATTN);
  // blocks in descending order: a document's later blocks see more keys, so
  // the longest CTAs launch first and the last wave holds the shortest
  const int split = blockIdx.x, g = blockIdx.y, blk = gridDim.z - 1 - blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // block table, positions and page table are written before the pass
  const int4 bd = p.blocks[blk];
  const int row0 = bd.x, nrows = bd.y, kmax = bd.z;
  const int mq = nrows * p.grp;
  // the block's document: its page table, page pool and TMA view
  const int32_t *table = p.views ? p.views[bd.w].table : p.table;
  const __nv_bfloat16 *pages =
      p.views ? (const __nv_bfloat16 *)p.views[bd.w].pages : p.pages;
  const CUtensorMap *tmap = p.tmaps ? p.tmaps + bd.w : &tm_kv;
  const int n_chunks = kmax / CH + 1;
  const int cps = (n_chunks + p.n_splits - 1) / p.n_splits;
  const int c0 = split * cps, c1 = min(n_chunks, c0 + cps);
  if (c0 >= c1) {  // empty split: the combine skips it
    pdl_trigger();
    return;
  }
  const int nch = c1 - c0;
  const uint32_t base = (su32(smem_raw) + 1023u) & ~1023u;
  const uint32_t sKV = base;
  volatile int *abort_v = &abort_f;
  auto page_row = [&](int c, int kv) {  // first row of (chunk c, kv) in the pool's 2D view
    const long long pg = table[c];
    return (int)((((pg * p.L + p.layer) * 2 + kv) * p.G + g) * CH);
  };
  const bool rows_cached = nch <= 64;

  if (tid == 0) {
    for (int st = 0; st < KV_STAGES; ++st) {
      mbar_init(&kv_full[st], 1);
      mbar_init(&kv_empty[st], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_free[b], SOFTMAX_THREADS);
      mbar_init(&p_full[b], SOFTMAX_THREADS);
      mbar_init(&o_done[b], 1);
    }
    mbar_init(&q_full, SOFTMAX_THREADS);
    mbar_init(&drain_bar, 1);
    abort_f = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  for (int v = tid; v < QV; v += NT5) spos[v] = v < mq ? p.pos[row0 + v / p.grp] : -1;
  // pull this CTA's K and V pages into L2 while the RoPE kernel finishes --
  // when they are few (a split key range: the repair).  A prefill CTA walks up
  // to 64 chunks from key 0; prefetching them all (about 150 MB over a wave)
  // only queued ahead of its own loads: 16.3 -> 14.8 ms of attention per
  // prefill without it.
  constexpr int PREFETCH_MAX_CHUNKS = 16;
  for (int t = tid; t < 2 * nch; t += NT5) {
    const int i = t >> 1, kv = t & 1;
    const int row = page_row(c0 + i, kv);
    if (rows_cached) sprow[t] = row;
    const __nv_bfloat16 *pg = pages + (size_t)row * DH;
    if (nch <= PREFETCH_MAX_CHUNKS)
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(pg), "r"(TBYTES)
                   : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     su32(&tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  // dependents may launch once this CTA holds its TMEM
  pdl_trigger();

  if (warp == 0) {
    // ------------------------------------------------------------ TMA
    if (lane == 0) {
      // a tensor map in global memory is read through the tensor-map proxy
      if (p.tmaps)
        asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(tmap)
                     : "memory");
      tma_prefetch_desc(tmap);
      pdl_wait();
      ts.waited();
      int issued = 0;
      for (int i = 0; i < nch && !*abort_v; ++i) {
        const int b = i % KV_STAGES;
        if (i >= KV_STAGES &&
            !mbar_wait(&kv_empty[b], (i / KV_STAGES - 1) & 1, abort_v, p.dev_flag, 64))
          break;
        const uint32_t sk = sKV + b * KVBYTES, sv = sk + TBYTES;
        mbar_expect_tx(&kv_full[b], KVBYTES);
        const int rk = rows_cached ? sprow[2 * i] : page_row(c0 + i, 0);
        const int rv = rows_cached ? sprow[2 * i + 1] : page_row(c0 + i, 1);
        if (i == 0) trace_mark(1);
#pragma unroll
        for (int h = 0; h < HALVES; ++h) {
          tma_load_2d((void *)__cvta_shared_to_generic(sk + h * CH * 128), tmap, &kv_full[b],
                      h * 64, rk);
          tma_load_2d((void *)__cvta_shared_to_generic(sv + h * CH * 128), tmap, &kv_full[b],
                      h * 64, rv);
        }
        ++issued;
      }
      // copies in flight complete before the CTA may exit
      for (int i = issued > KV_STAGES ? issued - KV_STAGES : 0; i < issued; ++i)
        mbar_wait(&kv_full[i % KV_STAGES], (i / KV_STAGES) & 1, abort_v, p.dev_flag, 0, false);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16(QV, CH), id_o = idesc_bf16(QV, DH, 1);
      // This one thread's issue path bounds the chunk rate (it shares its SM
      // sub-partition with four softmax warps), so the shared-memory
      // descriptors are built once: a stage, a 64-wide column block or a
      // 16-key slice only moves the start address, the descriptor's low field
      // (address / 16; the operands lie below 256 KB, so the field never
      // carries).
      const uint64_t dk0 = sw128_desc(sKV), dv0 = sw128_desc_mn(sKV + TBYTES, CH * 128, 1024);
      bool ok = mbar_wait(&q_full, 0, abort_v, p.dev_flag, 65);
      auto issue_s = [&](int i) -> bool {
        const int b = i & 1, st = i % KV_STAGES;
        if (!mbar_wait(&kv_full[st], (i / KV_STAGES) & 1, abort_v, p.dev_flag, 66)) return false;
        if (i >= 2 && !mbar_wait(&s_free[b], ((i - 2) >> 1) & 1, abort_v, p.dev_flag, 67))
          return false;
        tc_fence_after();
        const uint64_t dk = dk0 + (uint64_t)((st * KVBYTES) >> 4);
        const uint32_t ts = tmem + b * CH;
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk)  // 16 elements of head_dim: 8 columns of Q
          mma_bf16_ts(ts, tmem + T_Q + kk * 8,
                      dk + (uint64_t)(((kk >> 2) * CH * 128 + (kk & 3) * 32) >> 4), id_s,
                      kk > 0 ? 1u : 0u);
        mma_commit(&s_full[b]);
        return true;
      };
      // S of chunk i + 2 is issued as soon as the softmax has taken S of chunk
      // i out of its buffer (early in chunk i), ahead of O += P V of chunk i,
      // which waits for the end of that softmax: so S is ready before the
      // softmax reaches it, and the chunk rate is the softmax's own.  Issued
      // after P V of chunk i instead, it came about 1 us after that P.
      if (ok) ok = issue_s(0);
      if (ok && nch > 1) ok = issue_s(1);
      for (int i = 0; i < nch && ok; ++i) {
        if (i + 2 < nch && !(ok = issue_s(i + 2))) break;
        if (!(ok = mbar_wait(&p_full[i & 1], (i >> 1) & 1, abort_v, p.dev_flag, 68))) break;
        tc_fence_after();
        const uint64_t dv = dv0 + (uint64_t)(((i % KV_STAGES) * KVBYTES) >> 4);
        const uint32_t tp = tmem + T_P + (i & 1) * (CH / 2), to = tmem + 2 * CH;
        const uint32_t acc0 = i > 0 ? 1u : 0u;
#pragma unroll
        for (int kk = 0; kk < CH / 16; ++kk) {
          // P: a TMEM lane per query vector, 16 keys in 8 columns.  V: keys
          // are the rows (K), head_dim runs along them (MN-major) in 64-wide
          // column blocks CH*128 bytes apart, 8-key groups 1024 bytes apart;
          // 16 keys are 2048 bytes.
          mma_bf16_ts(to, tp + kk * 8, dv + (uint64_t)((kk * 2048) >> 4), id_o,
                      kk > 0 ? 1u : acc0);
        }
        mma_commit(&o_done[i & 1]);
        mma_commit(&kv_empty[i % KV_STAGES]);
      }
      // every MMA issued here completes before TMEM is freed
      mma_commit(&drain_bar);
      mbar_wait(&drain_bar, 0, abort_v, p.dev_flag, 0, false);
    }
  } else {
    // ------------------------------------------------------------ softmax
    // Warps w, w + 4, ... share TMEM lane quarter w % 4: the same 32 query
    // vectors, keys (and O columns) split in SMW parts.  Their per-chunk
    // maxima meet at a named barrier of the quarter's warps, which all of them
    // reach on every iteration -- also after an abort, when they only skip
    // their work -- so it can never wait on a warp that has left.
    const int quarter = warp & 3;  // TMEM lanes 32 * quarter .. + 31
    const int part = (warp - 2) >> 2;
    const int v = quarter * 32 + lane;
    const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
    const int bar_id = 1 + quarter;
    auto quad_bar = [&]() {
      asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "n"(32 * SMW) : "memory");
    };
    pdl_wait();
    // this thread's part of the Q row (DH / SMW elements, zero past the
    // block's query vectors) into the TMEM lane of query vector v
    {
      constexpr int QW = DH / (2 * SMW);  // 32-bit words (columns) of this part
      const bool real = v < mq;
      const uint4 *src = (const uint4 *)(p.q + ((size_t)(row0 + (real ? v / p.grp : 0)) * p.H +
                                                g * p.grp + v % p.grp) * DH) +
                         part * (QW / 4);
      uint32_t w[QW];
#pragma unroll
      for (int k = 0; k < QW / 4; ++k) {
        const uint4 x = real ? src[k] : make_uint4(0u, 0u, 0u, 0u);
        w[4 * k] = x.x;
        w[4 * k + 1] = x.y;
        w[4 * k + 2] = x.z;
        w[4 * k + 3] = x.w;
      }
#pragma unroll
      for (int k = 0; k < QW / 8; ++k) tmem_st8_nowait(tl + T_Q + part * QW + k * 8, w + 8 * k);
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(&q_full);
      if (warp == 2 && lane == 0) trace_mark(2);
    }
    constexpr int HK = CH / SMW;  // keys of this thread per chunk
    constexpr int OC = DH / SMW;  // O columns of this thread
    const int pv = spos[v];
    float m = -INFINITY, l = 0.f;  // reference maximum, this part's sum of exponentials
    bool dead = false;             // warp-uniform: a wait ran out
    for (int i = 0; i < nch; ++i) {
      const int b = i & 1, key0 = (c0 + i) * CH + part * HK;
      uint32_t sr[HK];
      float mx = -INFINITY;
      // every key of this part is causal for every query vector of the warp:
      // the chunk needs no mask (all but the diagonal chunk of a block)
      const bool unmasked = __all_sync(0xffffffffu, key0 + HK - 1 <= pv);
      if (!dead) {
        dead = !__all_sync(0xffffffffu,
                           mbar_wait(&s_full[b], (i >> 1) & 1, abort_v, p.dev_flag, 69));
      }
      if (!dead) {
        tc_fence_after();
        if (i == 0 && warp == 2 && lane == 0) trace_mark(3);
        if constexpr (HK == 32)
          tmem_ld32_nowait(tl + b * CH + part * HK, sr);
        else
          tmem_ld16_nowait(tl + b * CH + part * HK, sr);
        tmem_wait_ld();
        tc_fence_before();
        mbar_arrive(&s_free[b]);  // S is in registers: the buffer may be refilled
        float t[HK];
        if (unmasked) {
#pragma unroll
          for (int j = 0; j < HK; ++j) {
            const float x = __uint_as_float(sr[j]) * p.qk_scale;
            sr[j] = __float_as_uint(x);
            t[j] = x;
          }
        } else {
#pragma unroll
          for (int j = 0; j < HK; ++j) {
            const float x = __uint_as_float(sr[j]) * p.qk_scale;
            sr[j] = __float_as_uint(x);
            t[j] = key0 + j <= pv ? x : -INFINITY;
          }
        }
#pragma unroll
        for (int w = HK / 2; w > 0; w >>= 1)
#pragma unroll
          for (int j = 0; j < w; ++j) t[j] = fmaxf(t[j], t[j + w]);
        mx = t[0];
        sx[b][part][v] = mx;
      }
      quad_bar();
      if (dead) continue;
#pragma unroll
      for (int o = 0; o < SMW; ++o) mx = fmaxf(mx, sx[b][o][v]);
      // O is exactly zero until the first unmasked key: no rescale then.
      // The reference is an integer (see the header).
      if (m == -INFINITY) m = ceilf(mx);
      const bool grow = mx > m + RESCALE_LOG2;
      if (__any_sync(0xffffffffu, grow)) {
        if (i > 0) {  // O += P V of the previous chunk has landed
          dead = !__all_sync(0xffffffffu, mbar_wait(&o_done[(i - 1) & 1], ((i - 1) >> 1) & 1,
                                                    abort_v, p.dev_flag, 70));
          if (dead) continue;
          tc_fence_after();
        }
        const float mn = ceilf(mx);
        const float alpha = grow ? ex2(m - mn) : 1.f;
#pragma unroll
        for (int q = 0; q < OC / 16; ++q) {  // this part's O columns
          float o[16];
          tmem_ld16(tl + 2 * CH + part * OC + q * 16, o);
#pragma unroll
          for (int j = 0; j < 16; ++j) o[j] *= alpha;
          tmem_st16(tl + 2 * CH + part * OC + q * 16, o);
        }
        l *= alpha;
        if (grow) m = mn;
      }
      // P buffer b was last read by O += P V of chunk i - 2
      if (i >= 2) {
        dead = !__all_sync(0xffffffffu, mbar_wait(&o_done[b], ((i - 2) >> 1) & 1, abort_v,
                                                  p.dev_flag, 72));
        if (dead) continue;
      }
      float e[HK];
      if (unmasked) {
#pragma unroll
        for (int j = 0; j < HK; ++j) e[j] = ex2(__uint_as_float(sr[j]) - m);
      } else {
#pragma unroll
        for (int j = 0; j < HK; ++j) e[j] = key0 + j <= pv ? ex2(__uint_as_float(sr[j]) - m) : 0.f;
      }
      {  // P in bf16 pairs: this part's HK keys are HK / 2 columns of buffer b
        uint32_t w[HK / 2];
#pragma unroll
        for (int j = 0; j < HK / 2; ++j) w[j] = pack2(e[2 * j], e[2 * j + 1]);
#pragma unroll
        for (int q = 0; q < HK / 16; ++q)
          tmem_st8_nowait(tl + T_P + b * (CH / 2) + part * (HK / 2) + q * 8, w + 8 * q);
      }
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(&p_full[b]);
#pragma unroll
      for (int w = HK / 2; w > 0; w >>= 1)
#pragma unroll
        for (int j = 0; j < w; ++j) e[j] += e[j + w];
      l += e[0];
      if (warp == 2 && lane == 0) trace_mark(i == 0 ? 4 : 5);
    }
    if (!dead)
      dead = !__all_sync(0xffffffffu, mbar_wait(&o_done[(nch - 1) & 1], ((nch - 1) >> 1) & 1,
                                                abort_v, p.dev_flag, 71));
    if (warp == 2 && lane == 0) trace_mark(6);
    ssum[part][v] = l;
    quad_bar();
    float lt = 0.f;  // all parts, same reference maximum, summed in part order
#pragma unroll
    for (int o = 0; o < SMW; ++o) lt += ssum[o][v];
    // O: TMEM -> registers -> shared memory (the K/V stages are free now; rows
    // of DH floats, 16-byte chunks XOR-swizzled by row so the writes hit
    // distinct banks) -> global, one coalesced row per warp instruction.
    // Both named barriers are reached by all 256 softmax threads, live or not.
    constexpr int RCH = DH / 4;  // 16-byte chunks per staged row
    const float inv = lt > 0.f ? 1.f / lt : 0.f;
    const float scale = p.n_splits == 1 ? inv : 1.f;
    float *stage = (float *)__cvta_shared_to_generic(sKV);
    if (!dead) {
      tc_fence_after();
      const uint32_t to = tl + 2 * CH + part * OC;
      uint32_t o[OC];
      if constexpr (OC == 64) {
        tmem_ld32_nowait(to, o);
        tmem_ld32_nowait(to + 32, o + 32);
      } else if constexpr (OC == 32) {
        tmem_ld32_nowait(to, o);
      } else {
        tmem_ld16_nowait(to, o);
      }
      tmem_wait_ld();
      if (warp == 2 && lane == 0) trace_mark(7);
#pragma unroll
      for (int k = 0; k < OC / 4; ++k) {  // this part's chunks
        const int c = part * (OC / 4) + k;
        *(float4 *)(stage + v * DH + ((c ^ (v & (RCH - 1))) << 2)) =
            make_float4(__uint_as_float(o[4 * k]) * scale, __uint_as_float(o[4 * k + 1]) * scale,
                        __uint_as_float(o[4 * k + 2]) * scale, __uint_as_float(o[4 * k + 3]) * scale);
      }
      if (part == 0 && p.n_splits > 1 && v < mq) {
        const size_t bs = ((size_t)split * p.n_blocks + blk) * p.G + g;
        p.ws_ml[bs * WS_MAXQ + v] = make_float2(m, lt);
      }
    }
    asm volatile("bar.sync 5, %0;" ::"n"(SOFTMAX_THREADS) : "memory");
    {
      constexpr int RPW = QV / (4 * SMW);  // rows per softmax warp
      const int ws = warp - 2;             // rows ws * RPW .. + RPW - 1
      for (int rr = 0; rr < RPW; ++rr) {
        const int row = ws * RPW + rr;
        if (row >= mq || lane >= RCH) continue;
        const float4 x = *(const float4 *)(stage + row * DH + ((lane ^ (row & (RCH - 1))) << 2));
        if (p.n_splits == 1) {
          const int r = row0 + row / p.grp, hh = g * p.grp + row % p.grp;
          uint2 y;
          y.x = pack2(x.x, x.y);
          y.y = pack2(x.z, x.w);
          *(uint2 *)(p.out + ((size_t)r * p.H + hh) * DH + lane * 4) = y;
        } else {
          const size_t bs = ((size_t)split * p.n_blocks + blk) * p.G + g;
          *(float4 *)(p.ws_o + (bs * WS_MAXQ + row) * DH + lane * 4) = x;
        }
      }
    }
    if (warp == 2 && lane == 0) trace_mark(0);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(TMEM_COLS)
                 : "memory");
  ts.finish();
}

template <int DH>
constexpr size_t smem_bytes() {
  return 1024 + KV_STAGES * 2 * (size_t)CH * 128 * (DH / 64);
}

template <int DH>
const char *run(const CUtensorMap &tm, const Attn5Params &p, cudaStream_t s) {
  constexpr size_t smem = smem_bytes<DH>();
  static bool set = false;
  if (!set) {
    cudaError_t e = cudaFuncSetAttribute(k_attn_tc5<DH>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cudaGetErrorString(e);
    set = true;
  }
  dim3 grid(p.n_splits, p.G, p.n_blocks);
  launch_pdl(k_attn_tc5<DH>, grid, NT5, smem, s, tm, p);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

}  // namespace

int attn_tc5_rows_per_block(int grp) { return grp <= QV ? QV / grp : 0; }

// A CTA allocates all 512 tensor-memory columns of its SM.
int attn_tc5_ctas_per_sm(int) { return 1; }

const char *launch_attention_tc5(const void *q, const int32_t *pos, const int4 *blocks,
                                 int n_blocks, int n_splits, const Dims &dm, int layer,
                                 const void *pages, const int32_t *table, const CUtensorMap &tm_kv,
                                 float *ws_o, float2 *ws_ml, void *out, int *dev_flag,
                                 cudaStream_t s, const KVView *views,
                                 const CUtensorMap *tmaps) {
  if (n_blocks <= 0) return nullptr;
  if ((views == nullptr) != (tmaps == nullptr)) return "document views without tensor maps";
  Attn5Params p{};
  p.views = views;
  p.tmaps = tmaps;
  p.q = (const __nv_bfloat16 *)q;
  p.qk_scale = (float)(1.4426950408889634 / std::sqrt((double)dm.dh));
  p.pos = pos;
  p.blocks = blocks;
  p.pages = (const __nv_bfloat16 *)pages;
  p.table = table;
  p.H = dm.H;
  p.G = dm.G;
  p.grp = dm.H / dm.G;
  p.layer = layer;
  p.L = dm.L;
  p.n_splits = n_splits;
  p.n_blocks = n_blocks;
  p.ws_o = ws_o;
  p.ws_ml = ws_ml;
  p.out = (__nv_bfloat16 *)out;
  p.dev_flag = dev_flag;
  if (dm.dh == 128) return run<128>(tm_kv, p, s);
  if (dm.dh == 64) return run<64>(tm_kv, p, s);
  return "head_dim not supported";
}

KVR_TRACE_ATTACH(trace_attach_attn5)

}  // namespace kvr
