// k_gemm_tc.cu -- bf16 tensor-core GEMM for sm_103a: tcgen05.mma with TMEM
// accumulators, operands staged by TMA into 128B-swizzled shared memory.
//
//   Y[M][N] (+)= X[M][K] . W[N][K]^T     (bf16 operands, fp32 accumulate)
//
// Swap-AB: the weight W is the MMA's A operand (128 output features per tile
// = UMMA M), the M activation rows are its N dimension (BN <= 256 per tile),
// so a repair pass of ~40 rows still runs 128-row tensor-core tiles and the
// kernel streams W once from HBM.
//
// Work decomposition: persistent stream-K.  The units (feature tile, token
// tile, 64-wide K block) are linearised feature-tile-major and split into
// `grid` contiguous, equal ranges, one per CTA (grid <= #SMs), so every SM
// streams the same number of weight bytes whatever the GEMM shape.  A tile
// covered by several CTAs is either left to the kernel that next reads Y
// (deferred mode: each CTA stores its fp32 part and exits), or reduced here
// by its first CTA, for which it is the last segment: the others store their
// parts and publish them, the owner waits for them (bounded) and sums all
// parts in CTA order.  Either way the result is deterministic.
//
// Few-row GEMMs whose tiles cannot fill the GPU (e.g. O with 32 tiles) run
// in cluster split-K mode instead: the P CTAs of a thread-block cluster
// share one tile, each owning K/P of it; at the end each stages its partial
// tile in shared memory and, after a cluster barrier, sums its share of the
// rows over all P partials through distributed shared memory (rank order,
// deterministic) and applies the epilogue.  No global partials, fences or
// atomics on the tail.
//
// Warp roles (192 threads): warp 0 issues TMA loads (one elected lane), warp 1
// issues tcgen05.mma (one elected lane), warps 2-5 drain TMEM and run the
// epilogue.  Accumulators are double-buffered in TMEM so the MMA warp starts
// the next segment while the epilogue drains the previous one.
//
// Every mbarrier wait is bounded: a wait that runs out sets the device error
// flag and an abort flag in shared memory; all roles then stop issuing work,
// wait (bounded) for their copies and MMAs in flight, free TMEM and return.
#include <cooperative_groups.h>
#include <cstdlib>
#include <cuda.h>

#include "kvr_internal.cuh"
#include "tc_ptx.cuh"

namespace kvr {
namespace {
using namespace ptx;

constexpr int BM = 128;             // output features per tile (UMMA M)
constexpr int BK = 64;              // K per stage: one 128-byte swizzle atom of bf16
constexpr int UK = 16;              // K per tcgen05.mma kind::f16
// Epilogue warp groups: each group's four warps cover the four TMEM lane
// quarters (all 128 features of a tile); group e takes the 16-row chunks
// e, e + EPI_GROUPS, ... of a tile, so its chunks run in parallel.
constexpr int EPI_GROUPS = 2;
constexpr int EPI_THREADS = 128 * EPI_GROUPS;
constexpr int NTHREADS = 64 + EPI_THREADS;
constexpr int A_BYTES = BM * BK * 2;  // 16 KB
// Weight stages requested before the wait on the previous kernel.  All CTAs
// issue them at once into the same HBM queue; with the full pipeline (8) a CTA
// that becomes resident late waits behind every other CTA's deep prefetch for
// its first stage, and its whole range ends late.
constexpr int PRE_WAIT_STAGES = 4;

struct TcParams {
  int M, N, K;
  int BN, n_tiles, m_tiles, KB;
  int brows;  // rows of the activation TMA box: min(BN, M)
  long long total;
  int grid, stages;
  uint32_t tmem_cols;  // columns of one accumulator buffer
  float *Y;
  int ldy;
  const float *bias;
  int epi;
  void *out2;  // SwiGLU output (bf16 [M][N/2])
  int ld2;
  float *ws;        // [grid][2][BN][128] fp32 partial tiles
  int *counters;    // [2][max_tiles]: unused, then published parts per split tile (self-resetting)
  long long max_tiles;
  int *dev_flag;
  int cluster;  // > 1: cluster split-K with this many CTAs per tile
  int defer;    // 1: split tiles are left as partials for the consumer
  int stream_w; // 1: each weight tile is read once (one token tile): L2 evict-first
  // grouped data-parallel mode (dp_groups > 0, many rows): grid = dp_groups x
  // m_tiles CTAs; CTA i owns whole tiles -- token tile i % m_tiles of the
  // feature tiles dp_first(j) .. dp_first(j + 1) - 1 of group j = i / m_tiles
  // -- so the m_tiles CTAs of a group walk the same weight tiles in step and
  // read each from DRAM once.
  int dp_groups;
};

// First feature tile of data-parallel group j: groups take n_tiles / groups
// tiles, rounded down or up.
__device__ __forceinline__ int dp_first(const TcParams &p, int j) {
  return (int)((long long)j * p.n_tiles / p.dp_groups);
}

// ------------------------------------------------------------ PTX wrappers

__device__ __forceinline__ void epi_bar() {
  asm volatile("bar.sync 1, %0;" ::"n"(EPI_THREADS) : "memory");
}

// ------------------------------------------------------------ work split

// Units [a, b) of CTA i: stream-K ranges, or K/P of tile i/P in cluster mode
__device__ __forceinline__ void unit_range(long long i, long long total, int grid, int KB,
                                           int cluster, long long &a, long long &b) {
  if (cluster > 1) {
    long long tile = i / cluster, r = i % cluster;
    a = tile * KB + r * KB / cluster;
    b = tile * KB + (r + 1) * KB / cluster;
  } else {
    a = range_start(i, total, grid);
    b = range_start(i + 1, total, grid);
  }
}


// Epilogue for 16 consecutive rows t0..t0+15 of Y (the first `cnt` valid) at
// feature n of W.  All lanes of the warp call it together (SwiGLU exchanges
// lanes); every load is issued before any dependent use, so the chunk costs
// one L2 round trip, not sixteen.
template <class P>
__device__ __forceinline__ void epilogue16(const P &p, int t0, int n, const float *v, int cnt) {
  if (p.epi == GEMM_EPI_SWIGLU) {
    // rows 32b..32b+15 of W are gate, 32b+16..32b+31 up, of features
    // 16b..16b+15; lane = n % 32.  Lanes r and r ^ 16 swap their values, so
    // both hold gate and up of feature r % 16; the low half then writes the
    // even rows and the high half the odd ones.
    const int r = n & 31, hi = r >> 4;
    float o[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) o[j] = __shfl_xor_sync(0xffffffffu, v[j], 16);
    __nv_bfloat16 *out = (__nv_bfloat16 *)p.out2 + (size_t)t0 * p.ld2 + (n >> 5) * 16 + (r & 15);
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      // low lanes hold gate in v, up in o; high lanes the reverse
      const float g = hi ? o[2 * jj + 1] : v[2 * jj], u = hi ? v[2 * jj + 1] : o[2 * jj];
      const int j = 2 * jj + hi;
      if (j < cnt) out[(size_t)j * p.ld2] = __float2bfloat16_rn(swiglu_bf16path(g, u));
    }
    return;
  }
  float *y = p.Y + (size_t)t0 * p.ldy + n;
  if (p.epi == GEMM_EPI_ACCUM) {
    float old[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) old[j] = j < cnt ? y[(size_t)j * p.ldy] : 0.f;
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (j < cnt) y[(size_t)j * p.ldy] = old[j] + v[j];
    return;
  }
  float b = p.bias ? p.bias[n] : 0.f;
#pragma unroll
  for (int j = 0; j < 16; ++j)
    if (j < cnt) y[(size_t)j * p.ldy] = v[j] + b;
}

// The MMAs of units [u0, u1) of one GEMM: one TMEM accumulator per
// (feature tile, token tile) segment, double-buffered (seg counts segments);
// stage s / phase ph continue from the caller.  False if a wait ran out.
template <class P>
__device__ __forceinline__ bool mma_range(const P &p, long long u0, long long u1, int &s,
                                          uint32_t &ph, uint32_t &seg, int S, uint32_t base,
                                          uint32_t stage_bytes, uint32_t tmem_base,
                                          uint32_t idesc, uint64_t *full_bar, uint64_t *empty_bar,
                                          uint64_t *accf_bar, uint64_t *acce_bar,
                                          volatile int *abort_v) {
  bool ok = true;
  for (long long a = u0; a < u1 && ok;) {
    long long tl = a / p.KB;
    long long b = (tl + 1) * p.KB < u1 ? (tl + 1) * p.KB : u1;
    uint32_t buf = seg & 1u, use = seg >> 1;
    if (!mbar_wait(&acce_bar[buf], (use & 1u) ^ 1u, abort_v, p.dev_flag, 2)) break;
    tc_fence_after();
    uint32_t d = tmem_base + buf * p.tmem_cols;
    for (long long u = a; u < b; ++u) {
      if (!mbar_wait(&full_bar[s], ph, abort_v, p.dev_flag, 4)) {
        ok = false;
        break;
      }
      if (u == u0) trace_mark(0);
      tc_fence_after();
      uint32_t sa = base + (uint32_t)s * stage_bytes;
      uint64_t da = sw128_desc(sa), db = sw128_desc(sa + A_BYTES);
#pragma unroll
      for (int k = 0; k < BK / UK; ++k)
        mma_bf16(d, da + (uint64_t)(k * UK * 2 / 16), db + (uint64_t)(k * UK * 2 / 16), idesc,
                 (u > a || k > 0) ? 1u : 0u);
      mma_commit(&empty_bar[s]);
      if (++s == S) {
        s = 0;
        ph ^= 1u;
      }
    }
    if (ok) mma_commit(&accf_bar[buf]);
    ++seg;
    a = b;
  }
  return ok;
}

// The epilogue of units [u0, u1) of one GEMM (stream-K, one CTA's range):
// per segment, the accumulator from TMEM into Y (whole tiles), into the
// split-tile workspace (deferred mode), or, for a split tile's first CTA,
// summed with the other parts (bounded wait for them) in CTA order.
template <class P>
__device__ __forceinline__ void epi_range(const P &p, long long u0, long long u1, uint32_t &seg,
                                          uint32_t tmem_base, uint64_t *accf_bar,
                                          uint64_t *acce_bar, volatile int *abort_v, int q,
                                          int f, int et, int eg) {
  constexpr int CSTEP = 16 * EPI_GROUPS;
  for (long long a = u0; a < u1;) {
    long long tl = a / p.KB;
    long long b = (tl + 1) * p.KB < u1 ? (tl + 1) * p.KB : u1;
    uint32_t buf = seg & 1u, use = seg >> 1;
    int ntile = (int)(tl / p.m_tiles), mtile = (int)(tl % p.m_tiles);
    if (p.dp_groups) {  // a CTA-local tile of the grouped data-parallel mode
      ntile = dp_first(p, (int)(blockIdx.x / p.m_tiles)) + (int)tl;
      mtile = (int)(blockIdx.x % p.m_tiles);
    }
    int t0 = mtile * p.BN;
    int mv = min(p.BN, p.M - t0);
    int n = ntile * BM + f;
    long long tile_u0 = tl * p.KB;
    int i_first = p.dp_groups ? (int)blockIdx.x : cta_of(tile_u0, p.total, p.grid);
    int i_last = p.dp_groups ? (int)blockIdx.x : cta_of(tile_u0 + p.KB - 1, p.total, p.grid);
    int parts = i_last - i_first + 1;
    // The owner of a split tile waits for the other parts and, with two
    // parts and at most 48 rows, loads the other one now, while this
    // tile's MMAs are still running: both L2 round trips leave the tail.
    const bool own_fix = parts > 1 && !p.defer && (int)blockIdx.x == i_first;
    const bool pre = own_fix && parts == 2 && mv <= 48;
    // this group's chunks of the other part: chunk k of the group at rows
    // 16 eg + CSTEP k .. + 15
    constexpr int PRE_CHUNKS = (48 + CSTEP - 1) / CSTEP;
    float other[16 * PRE_CHUNKS];
    if (own_fix) {
      if (et == 0) {
        volatile int *ready = p.counters + p.max_tiles + tl;
        const uint64_t t0w = gtime_ns();
        for (uint32_t it = 0; *ready < parts - 1; ++it)
          if ((it & 63) == 63 && (*abort_v || gtime_ns() - t0w > WAIT_NS)) {
            if (!*abort_v) {
              *abort_v = 1;
              atomicOr(p.dev_flag, 32);
            }
            break;
          }
        trace_mark(4);
      }
      epi_bar();
      if (!*abort_v) {
        asm volatile("fence.acq_rel.gpu;" ::: "memory");  // acquire the parts
        if (pre) {
          const int so = range_start(i_last, p.total, p.grid) >= tile_u0 ? 0 : 1;
          const float *src = p.ws + ((size_t)i_last * 2 + so) * p.BN * BM + f;
#pragma unroll
          for (int k = 0; k < PRE_CHUNKS; ++k)
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int row = 16 * eg + CSTEP * k + j;
              other[16 * k + j] = row < mv ? __ldcg(src + (size_t)row * BM) : 0.f;
            }
        }
      }
    }
    if (!mbar_wait(&accf_bar[buf], use & 1u, abort_v, p.dev_flag, 8)) break;
    tc_fence_after();
    if (et == 0) trace_mark(2);
    uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + buf * p.tmem_cols;
    if (parts == 1) {
      for (int c = 16 * eg; c < mv; c += CSTEP) {
        float v[16];
        tmem_ld16(taddr + c, v);
        epilogue16(p, t0 + c, n, v, mv - c);
      }
      if (et == 0) trace_mark(5);
    } else if (p.defer) {
      // the consumer of Y adds this part: store it and go on
      int slot = range_start(blockIdx.x, p.total, p.grid) >= tile_u0 ? 0 : 1;
      float *w = p.ws + ((size_t)blockIdx.x * 2 + slot) * p.BN * BM;
      for (int c = 16 * eg; c < mv; c += CSTEP) {
        float v[16];
        tmem_ld16(taddr + c, v);
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (c + j < mv) w[(size_t)(c + j) * BM + f] = v[j];
      }
      if (et == 0) trace_mark(3);
    } else {
      // Reduced by its first CTA: for it the tile is the last segment, so
      // the others (for whom it is a first segment, or their whole range)
      // have usually published their parts long before.  A CTA that is not
      // the owner stores its part and publishes it; the owner keeps its own
      // part in TMEM, waits (bounded) until the others are published, and
      // sums all parts in CTA order.  Every CTA of the grid is resident (the
      // next kernel cannot launch before all of them have started) and a
      // publishing CTA waits on nothing, so the wait ends.
      const bool owner = (int)blockIdx.x == i_first;
      if (!owner) {
        int slot = range_start(blockIdx.x, p.total, p.grid) >= tile_u0 ? 0 : 1;
        float *w = p.ws + ((size_t)blockIdx.x * 2 + slot) * p.BN * BM;
        for (int c = 16 * eg; c < mv; c += CSTEP) {
          float v[16];
          tmem_ld16(taddr + c, v);
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (c + j < mv) w[(size_t)(c + j) * BM + f] = v[j];
        }
        asm volatile("fence.acq_rel.gpu;" ::: "memory");  // release the part
        epi_bar();
        if (et == 0) {
          atomicAdd(&p.counters[p.max_tiles + tl], 1);
          trace_mark(3);
        }
      } else {
        if (!*abort_v) {
#pragma unroll 1
          for (int c = 16 * eg; c < mv; c += CSTEP) {
            float own[16], v[16];
            tmem_ld16(taddr + c, own);
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] = 0.f;
            for (int i = i_first; i <= i_last; ++i) {
              if (i == (int)blockIdx.x) {
#pragma unroll
                for (int j = 0; j < 16; ++j) v[j] += own[j];
              } else if (pre) {
                // rows c..c+15 of the preloaded part: this group's chunk 0 or 1
                static_assert(PRE_CHUNKS == 2, "preloaded chunks of a group");
                const bool first = c == 16 * eg;
#pragma unroll
                for (int j = 0; j < 16; ++j) v[j] += first ? other[j] : other[16 + j];
              } else {
                const int si = range_start(i, p.total, p.grid) >= tile_u0 ? 0 : 1;
                const float *src = p.ws + (((size_t)i * 2 + si) * p.BN + c) * BM + f;
                float x[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) x[j] = c + j < mv ? __ldcg(src + (size_t)j * BM) : 0.f;
#pragma unroll
                for (int j = 0; j < 16; ++j) v[j] += x[j];
              }
            }
            epilogue16(p, t0 + c, n, v, mv - c);
          }
          if (et == 0) {
            p.counters[p.max_tiles + tl] = 0;
            trace_mark(5);
          }
        }
      }
    }
    tc_fence_before();
    mbar_arrive(&acce_bar[buf]);
    ++seg;
    a = b;
  }
}

__global__ void __launch_bounds__(NTHREADS, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
              const TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[8], empty_bar[8], accf_bar[2], acce_bar[2],
      drain_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_f;

  TraceScope ts(TK_GEMM);
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = p.stages;
  const uint32_t base = (su32(smem_raw) + 1023u) & ~1023u;
  const uint32_t stage_bytes = A_BYTES + (uint32_t)p.BN * 128u;
  const uint32_t tx_bytes = A_BYTES + (uint32_t)p.brows * 128u;
  long long u0, u1;
  if (p.dp_groups) {  // CTA-local units: the group's whole tiles
    const int j = (int)(blockIdx.x / p.m_tiles);
    u0 = 0;
    u1 = (long long)(dp_first(p, j + 1) - dp_first(p, j)) * p.KB;
  } else {
    unit_range(blockIdx.x, p.total, p.grid, p.KB, p.cluster, u0, u1);
  }

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf_bar[b], 1);
      mbar_init(&acce_bar[b], EPI_THREADS);
    }
    mbar_init(&drain_bar, 1);
    abort_f = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tmW);
      tma_prefetch_desc(&tmX);
    }
    __syncwarp();
    uint32_t ncols = 2 * p.tmem_cols;
    asm volatile(
        "tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
            su32(&tmem_slot)),
        "r"(ncols)
        : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_slot;
  volatile int *abort_v = &abort_f;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA
    if (lane == 0) {
      // incremental walk over (feature tile, token tile, K block) and stages
      long long tl0 = u0 / p.KB;
      int kb = (int)(u0 - tl0 * p.KB);
      int ntile = (int)(tl0 / p.m_tiles), mtile = (int)(tl0 - (long long)ntile * p.m_tiles);
      if (p.dp_groups) {
        ntile = dp_first(p, (int)(blockIdx.x / p.m_tiles));
        mtile = (int)(blockIdx.x % p.m_tiles);
      }
      const int mstep = p.dp_groups ? 0 : 1;  // the data-parallel walk keeps its token tile
      int s = 0;
      uint32_t ph = 0, it = 0;
      const uint64_t wpol = l2_evict_first();
      auto load_w = [&](uint32_t sa, uint64_t *bar, int x, int y) {
        if (p.stream_w)
          tma_load_2d_hint((void *)__cvta_shared_to_generic(sa), &tmW, bar, x, y, wpol);
        else
          tma_load_2d((void *)__cvta_shared_to_generic(sa), &tmW, bar, x, y);
      };
      // The weights never depend on the previous kernel: their tiles for the
      // first stages are requested before waiting for it (PDL), the
      // activation tiles of those stages right after.
      {
        const int pre_stages = S < PRE_WAIT_STAGES ? S : PRE_WAIT_STAGES;
        const long long npre = (u1 - u0) < pre_stages ? (u1 - u0) : pre_stages;
        int kb2 = kb, nt2 = ntile;
        int mt2 = mtile;
        for (long long j = 0; j < npre; ++j) {
          uint32_t sa = base + (uint32_t)j * stage_bytes;
          mbar_expect_tx(&full_bar[j], tx_bytes);
          load_w(sa, &full_bar[j], 0, (nt2 * p.KB + kb2) * BM);
          if (++kb2 == p.KB) {
            kb2 = 0;
            if ((mt2 += mstep) == p.m_tiles || !mstep) {
              mt2 = mstep ? 0 : mt2;
              ++nt2;
            }
          }
        }
        pdl_wait();
        ts.waited();
        for (long long j = 0; j < npre; ++j) {
          uint32_t sa = base + (uint32_t)j * stage_bytes;
          tma_load_2d((void *)__cvta_shared_to_generic(sa + A_BYTES), &tmX, &full_bar[j],
                      kb * BK, mtile * p.BN);
          ++it;
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
          if (++kb == p.KB) {
            kb = 0;
            if ((mtile += mstep) == p.m_tiles || !mstep) {
              mtile = mstep ? 0 : mtile;
              ++ntile;
            }
          }
        }
      }
      for (long long u = u0 + it; u < u1; ++u) {
        if (!mbar_wait(&empty_bar[s], ph ^ 1u, abort_v, p.dev_flag, 1)) break;
        uint32_t sa = base + (uint32_t)s * stage_bytes;
        mbar_expect_tx(&full_bar[s], tx_bytes);
        load_w(sa, &full_bar[s], 0, (ntile * p.KB + kb) * BM);
        tma_load_2d((void *)__cvta_shared_to_generic(sa + A_BYTES), &tmX, &full_bar[s], kb * BK,
                    mtile * p.BN);
        ++it;
        if (++s == S) {
          s = 0;
          ph ^= 1u;
        }
        if (++kb == p.KB) {
          kb = 0;
          if ((mtile += mstep) == p.m_tiles || !mstep) {
            mtile = mstep ? 0 : mtile;
            ++ntile;
          }
        }
      }
      // copies in flight complete before the CTA may exit
      uint32_t n_issued = it;
      for (uint32_t j = n_issued > (uint32_t)S ? n_issued - S : 0; j < n_issued; ++j)
        mbar_wait(&full_bar[j % S], (j / S) & 1u, abort_v, p.dev_flag, 0, false);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(BM, p.BN);
      uint32_t seg = 0, ph = 0;
      int s = 0;
      mma_range(p, u0, u1, s, ph, seg, S, base, stage_bytes, tmem_base, idesc, full_bar,
                empty_bar, accf_bar, acce_bar, abort_v);
      // all MMAs issued by this thread complete before TMEM is freed
      mma_commit(&drain_bar);
      mbar_wait(&drain_bar, 0, abort_v, p.dev_flag, 0, false);
      trace_mark(1);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    pdl_wait();  // outputs, partials and counters may still be in use upstream
    const int q = warp & 3;  // TMEM lane quarter of this warp
    const int f = q * 32 + lane;
    const int et = threadIdx.x - 64;  // 0 .. EPI_THREADS - 1
    const int eg = (warp - 2) >> 2;   // epilogue group: chunks 16 eg, 16 (eg + EPI_GROUPS), ...
    constexpr int CSTEP = 16 * EPI_GROUPS;
    uint32_t seg = 0;
    if (p.cluster > 1) {
      // stage this CTA's partial tile [mv][128] in shared memory (the
      // pipeline stages are free: every TMA load was consumed by the MMAs)
      if (mbar_wait(&accf_bar[0], 0, abort_v, p.dev_flag, 8)) {
        tc_fence_after();
        if (et == 0) trace_mark(2);
        const int mv = min(p.BN, p.M);
        float *sp = (float *)__cvta_shared_to_generic(base);
        uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16);
        for (int c = 16 * eg; c < mv; c += CSTEP) {
          float v[16];
          tmem_ld16(taddr + c, v);
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (c + j < mv) sp[(c + j) * BM + f] = v[j];
        }
        if (et == 0) trace_mark(3);
      }
      tc_fence_before();
    }
    if (p.cluster <= 1)
      epi_range(p, u0, u1, seg, tmem_base, accf_bar, acce_bar, abort_v, q, f, et, eg);
    if (et == 0) trace_mark(6);
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 64) trace_mark(7);
  if (p.cluster > 1) {
    // every CTA of the cluster reaches both barriers, on every path
    cooperative_groups::cluster_group cl = cooperative_groups::this_cluster();
    cl.sync();  // all partials staged
    if (threadIdx.x == 64) trace_mark(4);
    if (warp >= 2) {
      const int P = p.cluster, rank = (int)cl.block_rank();
      const int mv = min(p.BN, p.M);
      const int r0 = rank * mv / P, r1 = (rank + 1) * mv / P;
      const int f = (warp & 3) * 32 + lane;
      const int n = (int)(blockIdx.x / P) * BM + f;
      float *local = (float *)__cvta_shared_to_generic(base);
      for (int c = r0 + 16 * ((warp - 2) >> 2); c < r1; c += 16 * EPI_GROUPS) {
        float v[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] = 0.f;
        for (int qr = 0; qr < P; ++qr) {
          const float *rp = cl.map_shared_rank(local, qr);
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (c + j < r1) v[j] += rp[(c + j) * BM + f];
        }
        epilogue16(p, c, n, v, r1 - c);
      }
      if (threadIdx.x == 64) trace_mark(5);
    }
    cl.sync();  // peers have finished reading this CTA's shared memory
    if (threadIdx.x == 64) trace_mark(6);
  }
  tc_fence_after();
  if (warp == 0) {
    uint32_t ncols = 2 * p.tmem_cols;
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(ncols)
                 : "memory");
  }
  ts.finish();
}

// ------------------------------------------------------------ host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void *f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (EncodeTiledFn)f;
  }
  return fn;
}


// ------------------------------------------------------------ chained GEMMs
//
// A chain runs several GEMMs of one row set, with RMSNorms between them, in one
// persistent launch: the repair pass's O projection, RMSNorm, gate/up, down,
// the next layer's RMSNorm and QKV projection.  Every CTA keeps its pipeline,
// its TMEM and its role loops across the steps, and the steps meet at
// counters in device memory instead of kernel boundaries: the weight stream of
// the next GEMM starts while the last tiles of the previous one drain and
// while the norm runs (its weights do not depend on them), and no CTA leaves
// or is scheduled between steps.
//
// Step hand-offs (counters 128 bytes apart, zeroed before the pass):
//   after a GEMM, every CTA's epilogue, once its stores are done, adds one
//   behind a gpu-scope fence;
//   a norm (its row per CTA, CTAs 0 .. M-1) waits for all of them, completes
//   the GEMM's deferred split tiles into the residual, writes its row and adds
//   one;
//   a GEMM's TMA thread issues the first stages' weight tiles, waits for the
//   step before (the norm's M rows, or every CTA of the GEMM before) and only
//   then loads activations (after a generic-to-async proxy fence); its
//   epilogue waits for the same count before it writes outputs or split-tile
//   parts (the norm reads the previous GEMM's parts from the same workspace).
// All CTAs are resident at once (one per SM, grid = SM count, and the next
// kernel launches only after each has started), so every wait ends; each is
// bounded all the same.
constexpr int CHAIN_MAX = 6;         // steps per chain
constexpr int CHAIN_GEMMS = 4;       // GEMM steps per chain
constexpr int CHAIN_NORMS = 2;       // norm steps per chain
constexpr int CHAIN_BAR_STRIDE = 32;  // counters 128 bytes apart
constexpr int CHAIN_NORM_NV = 4;     // float4s per epilogue thread: d <= 4096

struct ChainNorm {
  float *h;            // [M][d] residual; split tiles of the GEMM before are added in place
  const float *g;      // [d] gains
  float eps;
  int d;               // multiple of 4, at most 4 * EPI_THREADS * CHAIN_NORM_NV
  __nv_bfloat16 *out;  // [M][d]
  SplitView sv;        // deferred split tiles of the GEMM before (ws null: none)
};

// Indexed by step.  The kernel takes it as a grid constant, so a step's fields
// are read in place from the parameter space (as an ordinary parameter,
// indexed by a run-time step, it was copied to local memory).
struct ChainParams {
  int n_steps, M;
  int is_norm[CHAIN_MAX];
  TcParams g[CHAIN_MAX];     // GEMM steps
  ChainNorm nrm[CHAIN_MAX];  // norm steps
  unsigned *bar;             // [CHAIN_MAX][CHAIN_BAR_STRIDE], zero at launch
  int *dev_flag;
};

struct ChainMaps {
  CUtensorMap w[CHAIN_MAX], x[CHAIN_MAX];  // GEMM steps
};

// Arrivals step k must see before it goes on: a norm's rows, or every CTA
// of a GEMM.
__device__ __forceinline__ unsigned chain_target(const ChainParams &c, int k) {
  return c.is_norm[k] ? (unsigned)c.M : (unsigned)c.g[k].grid;
}

// Bounded wait (2 s) until *ctr >= target: relaxed gpu-scope loads while it
// polls, then one acquire fence.
__device__ __forceinline__ bool chain_wait(const unsigned *ctr, unsigned target,
                                           volatile int *abort_f, int *dev_flag, int code) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
  if (v >= target) {
    asm volatile("fence.acq_rel.gpu;" ::: "memory");
    return true;
  }
  const uint64_t t0 = gtime_ns();
  for (uint32_t it = 0;; ++it) {
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
    if (v >= target) {
      asm volatile("fence.acq_rel.gpu;" ::: "memory");
      return true;
    }
    if ((it & 63) == 63) {
      if (*abort_f) return false;
      if (gtime_ns() - t0 > WAIT_NS) {
        *abort_f = 1;
        atomicOr(dev_flag, code);
        return false;
      }
    }
  }
}

__device__ __forceinline__ uint32_t chain_pack(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *(uint32_t *)&v;
}

// RMSNorm of residual row `row` by the CTA's EPI_THREADS epilogue threads
// (et = 0 .. EPI_THREADS - 1): the row, completed from the split view (and
// written back), normalised into out in bf16.  red: EPI_THREADS / 32 floats.
// The row's float4s are completed two at a time (each with up to
// SPLIT_MAX_PARTS part loads in flight): all four at once held too many
// registers for the kernel's budget.
__device__ __forceinline__ void chain_norm(const ChainNorm nm, int row, int et, float *red) {
  const int nq = nm.d >> 2;
  float4 *x = (float4 *)(nm.h + (size_t)row * nm.d);
  float4 v[CHAIN_NORM_NV];
  float ss = 0.f;
#pragma unroll 1
  for (int k0 = 0; k0 < CHAIN_NORM_NV; k0 += 2) {
#pragma unroll
    for (int k = k0; k < k0 + 2; ++k) {
      const int q = k * EPI_THREADS + et;
      float4 y = make_float4(0.f, 0.f, 0.f, 0.f);
      if (q < nq) {
        y = x[q];
        if (nm.sv.ws) {
          const SplitTile st =
              split_tile(nm.sv, (long long)(q >> 5) * nm.sv.m_tiles + row / nm.sv.BN);
          if (st.i0 != st.i1) {
            y = split_value4(nm.sv, st, y, row, 4 * q);
            x[q] = y;
          }
        }
      }
      ss += y.x * y.x + y.y * y.y + y.z * y.z + y.w * y.w;
      v[k] = y;
    }
  }
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((et & 31) == 0) red[et >> 5] = ss;
  epi_bar();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < EPI_THREADS / 32; ++w) tot += red[w];
  const float r = 1.0f / sqrtf(tot / (float)nm.d + nm.eps);
#pragma unroll
  for (int k = 0; k < CHAIN_NORM_NV; ++k) {
    const int q = k * EPI_THREADS + et;
    if (q < nq) {
      const float4 w = ((const float4 *)nm.g)[q];
      __nv_bfloat16 *o = nm.out + (size_t)row * nm.d + 4 * q;
      *(uint2 *)o = make_uint2(chain_pack(v[k].x * r * w.x, v[k].y * r * w.y),
                               chain_pack(v[k].z * r * w.z, v[k].w * r * w.w));
    }
  }
}

__global__ void __launch_bounds__(NTHREADS, 1)
    k_gemm_chain(const __grid_constant__ ChainMaps maps, const __grid_constant__ ChainParams c) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[8], empty_bar[8], accf_bar[2], acce_bar[2],
      drain_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_f;
  __shared__ float red[EPI_THREADS / 32];

  TraceScope ts(TK_GEMM);
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // every GEMM of a chain has the chain's rows: the same token tile, stage
  // layout, pipeline depth and accumulator width
  const TcParams &g0 = c.g[c.is_norm[0] ? 1 : 0];
  const int S = g0.stages;
  const uint32_t base = (su32(smem_raw) + 1023u) & ~1023u;
  const uint32_t stage_bytes = A_BYTES + (uint32_t)g0.BN * 128u;
  const uint32_t tx_bytes = A_BYTES + (uint32_t)g0.brows * 128u;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf_bar[b], 1);
      mbar_init(&acce_bar[b], EPI_THREADS);
    }
    mbar_init(&drain_bar, 1);
    abort_f = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    if (lane < c.n_steps && !c.is_norm[lane]) {
      tma_prefetch_desc(&maps.w[lane]);
      tma_prefetch_desc(&maps.x[lane]);
    }
    __syncwarp();
    uint32_t ncols = 2 * g0.tmem_cols;
    asm volatile(
        "tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
            su32(&tmem_slot)),
        "r"(ncols)
        : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_slot;
  volatile int *abort_v = &abort_f;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0, it = 0;
      const uint64_t wpol = l2_evict_first();
#pragma unroll 1
      for (int k = 0; k < CHAIN_MAX; ++k) {
        if (k >= c.n_steps || *abort_v) break;
        if (c.is_norm[k]) continue;
        const TcParams &p = c.g[k];
        const CUtensorMap *tW = &maps.w[k], *tX = &maps.x[k];
        long long u0, u1;
        unit_range(blockIdx.x, p.total, p.grid, p.KB, 0, u0, u1);
        long long tl0 = u0 / p.KB;
        int kb = (int)(u0 - tl0 * p.KB);
        int ntile = (int)(tl0 / p.m_tiles), mtile = (int)(tl0 - (long long)ntile * p.m_tiles);
        auto advance = [&]() {
          ++it;
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
          if (++kb == p.KB) {
            kb = 0;
            if (++mtile == p.m_tiles) {
              mtile = 0;
              ++ntile;
            }
          }
        };
        auto load_w = [&](uint32_t sa) {
          const int y = (ntile * p.KB + kb) * BM;
          if (p.stream_w)
            tma_load_2d_hint((void *)__cvta_shared_to_generic(sa), tW, &full_bar[s], 0, y, wpol);
          else
            tma_load_2d((void *)__cvta_shared_to_generic(sa), tW, &full_bar[s], 0, y);
        };
        // the first stages' weights before the step's input is ready
        const long long npre = (u1 - u0) < S ? (u1 - u0) : S;
        int pre_s[8], pre_kb[8], pre_mt[8];
        long long u = u0;
        for (; u < u0 + npre; ++u) {
          if (!mbar_wait(&empty_bar[s], ph ^ 1u, abort_v, c.dev_flag, 1)) break;
          const uint32_t sa = base + (uint32_t)s * stage_bytes;
          mbar_expect_tx(&full_bar[s], tx_bytes);
          load_w(sa);
          pre_s[u - u0] = s;
          pre_kb[u - u0] = kb;
          pre_mt[u - u0] = mtile;
          advance();
        }
        const int npre_done = (int)(u - u0);
        bool ready = true;
        if (k == 0) {
          pdl_wait();
        } else {
          ready = chain_wait(c.bar + (size_t)(k - 1) * CHAIN_BAR_STRIDE, chain_target(c, k - 1),
                             abort_v, c.dev_flag, 80 + k);
          // the input was written by generic stores; TMA reads it
          asm volatile("fence.proxy.async.global;" ::: "memory");
        }
        if (k == 0) ts.waited();
        // the activations of the stages begun (read even after a wait ran
        // out, so that every stage's transaction completes)
        for (int j = 0; j < npre_done; ++j) {
          const uint32_t sa = base + (uint32_t)pre_s[j] * stage_bytes;
          tma_load_2d((void *)__cvta_shared_to_generic(sa + A_BYTES), tX, &full_bar[pre_s[j]],
                      pre_kb[j] * BK, pre_mt[j] * p.BN);
        }
        if (!ready || npre_done < npre) break;
        for (; u < u1; ++u) {
          if (!mbar_wait(&empty_bar[s], ph ^ 1u, abort_v, c.dev_flag, 1)) break;
          const uint32_t sa = base + (uint32_t)s * stage_bytes;
          mbar_expect_tx(&full_bar[s], tx_bytes);
          load_w(sa);
          tma_load_2d((void *)__cvta_shared_to_generic(sa + A_BYTES), tX, &full_bar[s], kb * BK,
                      mtile * p.BN);
          advance();
        }
      }
      // copies in flight complete before the CTA may exit
      for (uint32_t j = it > (uint32_t)S ? it - S : 0; j < it; ++j)
        mbar_wait(&full_bar[j % S], (j / S) & 1u, abort_v, c.dev_flag, 0, false);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(BM, g0.BN);
      uint32_t seg = 0, ph = 0;
      int s = 0;
#pragma unroll 1
      for (int k = 0; k < CHAIN_MAX; ++k) {
        if (k >= c.n_steps) break;
        if (c.is_norm[k]) continue;
        const TcParams &p = c.g[k];
        long long u0, u1;
        unit_range(blockIdx.x, p.total, p.grid, p.KB, 0, u0, u1);
        if (!mma_range(p, u0, u1, s, ph, seg, S, base, stage_bytes, tmem_base, idesc, full_bar,
                       empty_bar, accf_bar, acce_bar, abort_v))
          break;
      }
      // all MMAs issued by this thread complete before TMEM is freed
      mma_commit(&drain_bar);
      mbar_wait(&drain_bar, 0, abort_v, c.dev_flag, 0, false);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;  // TMEM lane quarter of this warp
    const int f = q * 32 + lane;
    const int et = threadIdx.x - 64;  // 0 .. EPI_THREADS - 1
    const int eg = (warp - 2) >> 2;   // epilogue group
    uint32_t seg = 0;
#pragma unroll 1
    for (int k = 0; k < CHAIN_MAX; ++k) {
      if (k >= c.n_steps) break;
      unsigned *arrive = c.bar + (size_t)k * CHAIN_BAR_STRIDE;
      if (!c.is_norm[k]) {
        // the step before is done before outputs or parts are written:
        // the norm before reads the workspace this GEMM's parts go to
        if (k == 0) {
          pdl_wait();
        } else {
          if (et == 0)
            chain_wait(c.bar + (size_t)(k - 1) * CHAIN_BAR_STRIDE, chain_target(c, k - 1),
                       abort_v, c.dev_flag, 90 + k);
          epi_bar();
        }
        const TcParams &p = c.g[k];
        long long u0, u1;
        unit_range(blockIdx.x, p.total, p.grid, p.KB, 0, u0, u1);
        epi_range(p, u0, u1, seg, tmem_base, accf_bar, acce_bar, abort_v, q, f, et, eg);
        epi_bar();  // every store of the step is issued by now
        if (et == 0) {
          __threadfence();
          atomicAdd(arrive, 1u);
        }
      } else if ((int)blockIdx.x < c.M) {
        if (k == 0) {
          pdl_wait();
        } else {
          if (et == 0)
            chain_wait(c.bar + (size_t)(k - 1) * CHAIN_BAR_STRIDE, chain_target(c, k - 1),
                       abort_v, c.dev_flag, 90 + k);
          epi_bar();
        }
        chain_norm(c.nrm[k], blockIdx.x, et, red);
        epi_bar();
        if (et == 0) {
          __threadfence();
          atomicAdd(arrive, 1u);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) {
    uint32_t ncols = 2 * g0.tmem_cols;
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(ncols)
                 : "memory");
  }
  ts.finish();
}

}  // namespace

// The weight in the blocked layout (make_tmap_weight): 8 bf16 (one uint4) at a
// time, row-major element (n, k) <-> block (n / 128, k / 64), row n % 128,
// column k % 64.
__global__ void k_weight_tile(const uint4 *src, uint4 *dst, int N, int K, int untile) {
  const int K8 = K / 8, KB = K / BK;
  const long long total = (long long)N * K8;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int n = (int)(e / K8), k = (int)(e % K8) * 8;
    const long long t =
        (((long long)(n / BM) * KB + k / BK) * BM + n % BM) * (BK / 8) + (k % BK) / 8;
    if (untile)
      dst[e] = src[t];
    else
      dst[t] = src[e];
  }
}

bool make_tmap_bf16(CUtensorMap *map, const void *ptr, int rows, int cols, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || ((uintptr_t)ptr & 15) || (cols * 2) % 16 || box_rows > 256 || box_rows < 1)
    return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {BK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims,
                  strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool gemm_tc_supported(int N, int K) { return N % BM == 0 && K % BK == 0 && N > 0 && K > 0; }

bool make_tmap_weight(CUtensorMap *map, const void *w, int N, int K) {
  if (!gemm_tc_supported(N, K)) return false;
  const long long rows = (long long)N * K / BK;
  return rows < (1ll << 31) && make_tmap_bf16(map, w, (int)rows, BK, BM);
}

const char *launch_weight_tile(const void *src, void *dst, int N, int K, bool untile,
                               cudaStream_t s) {
  if (!gemm_tc_supported(N, K)) return "weight shape not tiled";
  const long long n = (long long)N * K / 8;
  const int grid = (int)std::min<long long>((n + 255) / 256, 65536);
  k_weight_tile<<<grid, 256, 0, s>>>((const uint4 *)src, (uint4 *)dst, N, K, untile ? 1 : 0);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

namespace {
// Cluster split-K width for a few-row GEMM whose n_tiles cannot fill the
// SMs: the largest P <= 8 with n_tiles * P <= #SMs, used when it covers at
// least 3/4 of the SMs and all clusters fit in one wave; else 0 (stream-K).
int choose_cluster(int M, int N, int num_sms, size_t smem) {
  static const bool off = [] {
    const char *e = getenv("KVR_DISABLE_CLUSTER_SPLITK");
    return e && e[0] == '1';
  }();
  if (off || M > 64) return 0;
  int T = N / BM;
  int P = num_sms / T;
  if (P > 8) P = 8;
  if (P < 2 || T * P * 4 < num_sms * 3) return 0;
  static int cache_p[16] = {0}, cache_ok[16] = {0};
  static size_t cache_smem[16] = {0};
  for (int i = 0; i < 16; ++i)
    if (cache_p[i] == P && cache_smem[i] == smem) return cache_ok[i] >= T ? P : 0;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(T * P);
  cfg.blockDim = dim3(NTHREADS);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = P;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  int nc = 0;
  if (cudaOccupancyMaxActiveClusters(&nc, (void *)k_gemm_tc, &cfg) != cudaSuccess) {
    cudaGetLastError();
    nc = 0;
  }
  for (int i = 0; i < 16; ++i)
    if (cache_p[i] == 0) {
      cache_p[i] = P;
      cache_smem[i] = smem;
      cache_ok[i] = nc;
      break;
    }
  return nc >= T ? P : 0;
}
}  // namespace

int gemm_tc_bn(int M) {
  if (M > 256) return 256;
  int bn = (M + 15) / 16 * 16;
  return bn < 16 ? 16 : bn;
}

size_t gemm_tc_ws_bytes(int num_sms) { return (size_t)num_sms * 2 * 256 * BM * sizeof(float); }

namespace {

// Dynamic shared memory this kernel may use (opt-in limit minus static);
// < 0 on failure.
int dyn_smem_limit() {
  static int max_dyn = -1;
  if (max_dyn < 0) {
    int dev = 0, optin = 0;
    cudaFuncAttributes fa{};
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (cudaFuncGetAttributes(&fa, k_gemm_tc) != cudaSuccess) return -1;
    int lim = optin - (int)fa.sharedSizeBytes;
    if (cudaFuncSetAttribute(k_gemm_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, lim) !=
        cudaSuccess)
      return -1;
    max_dyn = lim;
  }
  return max_dyn;
}

// Tiling, pipeline depth and split of an M x N x K GEMM: fills the shape
// fields of p and the dynamic shared memory; nullptr on success.
const char *configure(int M, int N, int K, int num_sms, bool defer, TcParams &p, size_t &smem) {
  p.M = M;
  p.N = N;
  p.K = K;
  p.BN = gemm_tc_bn(M);
  p.n_tiles = N / BM;
  p.m_tiles = (M + p.BN - 1) / p.BN;
  p.KB = K / BK;
  // A box may not be taller than the tensor: a single short token tile loads
  // just its M rows (the MMA's extra columns are never stored).
  p.brows = p.BN < M ? p.BN : M;
  p.total = (long long)p.n_tiles * p.m_tiles * p.KB;
  p.grid = (int)(p.total < num_sms ? p.total : num_sms);
  int max_dyn = dyn_smem_limit();
  if (max_dyn < 0) return "cannot raise the dynamic shared memory limit";
  uint32_t stage_bytes = A_BYTES + (uint32_t)p.BN * 128u;
  int smem_budget = max_dyn - 1024;
  p.stages = smem_budget / (int)stage_bytes;
  if (p.stages > 8) p.stages = 8;
  if (p.stages < 2) return "token tile too large for shared memory";
  uint32_t cols = 32;
  while (cols < (uint32_t)p.BN) cols <<= 1;
  p.tmem_cols = cols;
  smem = 1024 + (size_t)p.stages * stage_bytes;
  p.defer = defer ? 1 : 0;
  p.cluster = p.m_tiles == 1 && !defer ? choose_cluster(M, N, num_sms, smem) : 0;
  p.stream_w = p.m_tiles == 1;
  if (p.cluster > 1) p.grid = p.n_tiles * p.cluster;
  p.dp_groups = 0;
  // Many rows (a prefill chunk): the grouped data-parallel mode when some
  // token tile width and group count fill at least 90% of the SMs' slots with
  // useful work: rows over padded rows, CTAs over SMs, and a group's tiles
  // over the largest group's (groups need not divide the feature tiles).
  // Stream-K there walks all token tiles of a feature tile per CTA, so the
  // 152 CTAs' weights (about 1 MB each) overflow L2 and every weight tile
  // came from DRAM once per token tile.
  static const bool dp_off = [] {
    const char *e = getenv("KVR_DISABLE_DP_GEMM");
    return e && e[0] == '1';
  }();
  if (!dp_off && M >= 512) {
    double best = 0.0;
    int bbn = 0, bmt = 0, bg = 0;
    for (int bn = 256; bn >= 128; bn -= 16) {
      const int mt = (M + bn - 1) / bn;
      for (int g = 1; g <= p.n_tiles && g * mt <= num_sms; ++g) {
        const int most = (p.n_tiles + g - 1) / g;
        const double eff = (double)M / ((double)mt * bn) * (double)(g * mt) / num_sms *
                           ((double)p.n_tiles / g / most);
        if (eff > best + 1e-9) {
          best = eff;
          bbn = bn;
          bmt = mt;
          bg = g;
        }
      }
    }
    const uint32_t sb = A_BYTES + (uint32_t)bbn * 128u;
    const int st = bbn ? smem_budget / (int)sb : 0;
    if (best >= 0.9 && st >= 2) {
      p.BN = bbn;
      p.m_tiles = bmt;
      p.brows = bbn < M ? bbn : M;
      p.total = (long long)p.n_tiles * p.m_tiles * p.KB;
      p.grid = bg * bmt;
      p.dp_groups = bg;
      p.stages = st > 8 ? 8 : st;
      uint32_t c2 = 32;
      while (c2 < (uint32_t)p.BN) c2 <<= 1;
      p.tmem_cols = c2;
      smem = 1024 + (size_t)p.stages * sb;
      p.defer = 0;  // whole tiles: nothing is split
      p.cluster = 0;
      p.stream_w = 0;
    }
  }
  return nullptr;
}

}  // namespace

const char *launch_gemm_tc(const GemmArgs &g, const CUtensorMap &tmW, int epi, void *out2,
                           int ld2, const TcWorkspace &ws, cudaStream_t s, SplitView *defer) {
  if (defer) *defer = SplitView{};
  if (g.M <= 0) return nullptr;
  bool dfr = defer != nullptr && epi != GEMM_EPI_SWIGLU;
  TcParams p{};
  size_t smem = 0;
  if (const char *e = configure(g.M, g.N, g.K, ws.num_sms, dfr, p, smem)) return e;
  if (p.dp_groups) dfr = false;  // whole tiles per CTA: no split tiles to leave
  if (dfr) {
    // CTAs per tile: at most ceil(KB / (units per CTA)) + 1
    long long per = p.total / p.grid;
    if (per < 1 || (p.KB + per - 1) / per + 1 > SPLIT_MAX_PARTS) {
      dfr = false;
      if (const char *e = configure(g.M, g.N, g.K, ws.num_sms, false, p, smem)) return e;
    }
  }
  p.Y = g.Y;
  p.ldy = g.ldy;
  p.bias = g.bias;
  p.epi = epi;
  p.out2 = out2;
  p.ld2 = ld2;
  p.ws = ws.partials;
  p.counters = ws.counters;
  p.max_tiles = ws.max_tiles;
  p.dev_flag = ws.dev_flag;
  if ((long long)p.n_tiles * p.m_tiles > ws.max_tiles) return "more tiles than counters";
  CUtensorMap tmX;
  if (!make_tmap_bf16(&tmX, g.X, g.M, g.K, p.brows)) return "activation TMA descriptor rejected";
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(p.grid);
  cfg.blockDim = dim3(NTHREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  int na = 0;
  if (g_pdl) {
    at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  if (p.cluster > 1) {
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = p.cluster;
    at[na].val.clusterDim.y = 1;
    at[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = at;
  cfg.numAttrs = na;
  cudaLaunchKernelEx(&cfg, k_gemm_tc, tmW, tmX, p);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess && dfr) {
    // a tile is split when a range boundary falls inside it
    bool split = false;
    for (int i = 0; i < p.grid && !split; ++i)
      split = range_start(i, p.total, p.grid) % p.KB != 0;
    if (split) {
      defer->ws = ws.partials;
      defer->bias = epi == GEMM_EPI_STORE ? g.bias : nullptr;
      defer->total = p.total;
      defer->grid = p.grid;
      defer->KB = p.KB;
      defer->BN = p.BN;
      defer->m_tiles = p.m_tiles;
      defer->accum = epi == GEMM_EPI_ACCUM ? 1 : 0;
      defer->small = (p.total + 1) * (long long)p.grid < (1ll << 31) ? 1 : 0;
    }
  }
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

size_t gemm_chain_bar_words() { return (size_t)CHAIN_MAX * CHAIN_BAR_STRIDE; }

const char *launch_gemm_chain(const ChainStep *st, int n, const TcWorkspace &ws, unsigned *bar,
                              cudaStream_t s, SplitView *last_defer) {
  if (last_defer) *last_defer = SplitView{};
  if (n < 1 || n > CHAIN_MAX) return "chain length outside [1, 6]";
  ChainParams c{};
  ChainMaps maps{};
  c.n_steps = n;
  c.bar = bar;
  c.dev_flag = ws.dev_flag;
  int ng = 0, nn = 0, M = -1, first = -1;
  size_t smem = 0;
  SplitView prev{};  // deferred split tiles of the GEMM just before
  for (int k = 0; k < n; ++k) {
    c.is_norm[k] = st[k].norm ? 1 : 0;
    if (st[k].norm) {
      if (nn == CHAIN_NORMS) return "more than two norms in a chain";
      if (k + 1 < n && st[k + 1].norm) return "two norms in a row";
      ChainNorm &nm = c.nrm[k];
      nm.h = st[k].h;
      nm.g = st[k].gain;
      nm.eps = st[k].eps;
      nm.d = st[k].d;
      nm.out = (__nv_bfloat16 *)st[k].out;
      nm.sv = prev;
      if (nm.d % 4 || nm.d > 4 * EPI_THREADS * CHAIN_NORM_NV) return "norm width";
      if (((uintptr_t)nm.h | (uintptr_t)nm.g | (uintptr_t)nm.out) & 15) return "norm alignment";
      prev = SplitView{};
      ++nn;
      continue;
    }
    if (ng == CHAIN_GEMMS) return "more than four GEMMs in a chain";
    const GemmArgs &g = st[k].g;
    if (M < 0) M = g.M;
    if (g.M != M || g.M <= 0) return "chain GEMMs of different row counts";
    if (first < 0) first = k;
    TcParams &p = c.g[k];
    const bool dfr = st[k].defer && st[k].epi != GEMM_EPI_SWIGLU;
    size_t sm = 0;
    if (const char *e = configure(g.M, g.N, g.K, ws.num_sms, dfr, p, sm)) return e;
    if (p.dp_groups) return "chain GEMM with many rows (data-parallel tiling)";
    p.cluster = 0;  // stream-K over the whole grid
    p.grid = (int)(p.total < ws.num_sms ? p.total : ws.num_sms);
    if (p.grid != ws.num_sms) return "chain GEMM with fewer units than SMs";
    if (dfr) {
      const long long per = p.total / p.grid;
      if (per < 1 || (p.KB + per - 1) / per + 1 > SPLIT_MAX_PARTS) return "chain GEMM split too fine";
    }
    if ((long long)p.n_tiles * p.m_tiles > ws.max_tiles) return "more tiles than counters";
    if (first != k && (p.stages != c.g[first].stages || p.BN != c.g[first].BN))
      return "chain GEMMs of different tilings";
    p.Y = g.Y;
    p.ldy = g.ldy;
    p.bias = g.bias;
    p.epi = st[k].epi;
    p.out2 = st[k].out2;
    p.ld2 = st[k].ld2;
    p.ws = ws.partials;
    p.counters = ws.counters;
    p.max_tiles = ws.max_tiles;
    p.dev_flag = ws.dev_flag;
    maps.w[k] = *st[k].tmW;
    if (!make_tmap_bf16(&maps.x[k], g.X, g.M, g.K, p.brows))
      return "activation TMA descriptor rejected";
    smem = sm > smem ? sm : smem;
    prev = SplitView{};
    if (dfr) {
      bool split = false;
      for (int i = 0; i < p.grid && !split; ++i) split = range_start(i, p.total, p.grid) % p.KB != 0;
      if (split) {
        prev.ws = ws.partials;
        prev.bias = p.epi == GEMM_EPI_STORE ? g.bias : nullptr;
        prev.total = p.total;
        prev.grid = p.grid;
        prev.KB = p.KB;
        prev.BN = p.BN;
        prev.m_tiles = p.m_tiles;
        prev.accum = p.epi == GEMM_EPI_ACCUM ? 1 : 0;
        prev.small = (p.total + 1) * (long long)p.grid < (1ll << 31) ? 1 : 0;
      }
    }
    p.defer = dfr ? 1 : 0;
    ++ng;
  }
  if (ng == 0) return "chain without a GEMM";
  if (st[0].norm && (n < 2 || st[1].norm)) return "a chain's first norm feeds no GEMM";
  if (nn > 0 && M > ws.num_sms) return "chain norm rows above the SM count";
  c.M = M;
  static int set_smem = -1;
  if (set_smem < (int)smem) {
    cudaError_t e = cudaFuncSetAttribute(k_gemm_chain, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cudaGetErrorString(e);
    set_smem = (int)smem;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(ws.num_sms);
  cfg.blockDim = dim3(NTHREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = g_pdl ? 1 : 0;
  cudaLaunchKernelEx(&cfg, k_gemm_chain, maps, c);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cudaGetErrorString(e);
  if (last_defer) *last_defer = prev;
  return nullptr;
}

KVR_TRACE_ATTACH(trace_attach_gemm)

}  // namespace kvr
