// kvr_internal.cuh -- internal declarations of libkvrepair (not installed).
//
// Device data layout (HBM):
//   weights  one allocation; per layer
//              wqkv [(H+2G)*dh][d]   rows: q heads, then k heads, then v heads
//              bqkv fp32 [(H+2G)*dh] (QKV-bias models only)
//              wo   [d][H*dh]
//              wgu  [2F][d]          gate/up rows interleaved in blocks of 16:
//                                    rows 32b..32b+15 = gate 16b..16b+15,
//                                    rows 32b+16..32b+31 = up 16b..16b+15
//              wd   [d][F]
//              attn_norm, mlp_norm fp32 [d]
//            embed [V][d], lm_head [V][d], final_norm fp32 [d]
//   KV cache paged: page = KVR_PAGE positions of every layer,
//            [page][layer][k|v][kv head][slot][dh] in the model dtype;
//            a block table maps logical page -> physical page.
//   activations (per model workspace, max_rows R): residual h fp32 [R][d],
//            normed rows a [R][d], qkv fp32 [R][Nqkv], q fp32 [R][H*dh],
//            attention output [R][H*dh], gate/up fp32 [R][2F], act [R][F].
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <string>
#include <vector>

#include "../../include/kvrepair.h"

namespace kvr {

constexpr int KVR_PAGE = 64;          // positions per KV page
constexpr int KVR_RD_GROUPS = 8;      // layer groups of kvr_repair_read's overlapped copies
constexpr int KVR_QUERY_RESERVE = 64; // positions past n reserved for fresh queries
constexpr int GU_BLOCK = 16;          // gate/up interleave block (rows)

struct Dims {
  int V, d, L, H, G, dh, F;
  int qkv_bias, dtype, delim;
  double theta, eps;
  int max_ctx, max_rows;
  int Nqkv() const { return (H + 2 * G) * dh; }
  size_t es() const { return dtype == KVR_DTYPE_BF16 ? 2 : 4; }
  // elements of one KV page (all layers, k and v)
  size_t page_elems() const { return (size_t)L * 2 * G * KVR_PAGE * dh; }
};

struct LayerW {
  void *wqkv, *wo, *wgu, *wd;
  float *bqkv, *attn_norm, *mlp_norm;
  // TMA descriptors of the weights (bf16 models, tensor-core GEMM shapes)
  CUtensorMap tm_qkv, tm_o, tm_gu, tm_d;
  bool tc_qkv, tc_o, tc_gu, tc_d;
};

// Device view of one document's paged cache (passed by value to kernels).
struct KVView {
  void *pages;              // pool base
  const int32_t *table;     // logical page -> physical page
  int L, G, dh;             // shape
  __host__ __device__ size_t offset(int layer, int kv, int g, int pos) const {
    size_t page = (size_t)table[pos / KVR_PAGE];
    return ((((page * L + layer) * 2 + kv) * G + g) * KVR_PAGE + (pos % KVR_PAGE)) * dh;
  }
};

// Scratch of the tensor-core GEMM (split-tile partials, arrival counters).
// Device timeline trace buffer (see TraceScope).
struct TraceBuf {
  unsigned long long *rec = nullptr;
  unsigned int *count = nullptr;
  unsigned int cap = 0;
};

// silu(g) * u for the bf16 tensor-core GEMM's fused epilogue: g sigma(g) with
// sigma(g) = 1 / (1 + 2^(-g log2 e)) from the hardware base-2 exponential and
// reciprocal (relative error about 1e-7, so the bf16 rounding of the result is
// that of the exact product up to rare ties; the hardware tanh, one op fewer,
// is off by up to 1e-3, half a bf16 step).  Large |g| saturate to g or -0.
__device__ __forceinline__ float swiglu_bf16path(float g, float u) {
  float e, r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(-1.4426950408889634f * g));
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(1.0f + e));
  return g * r * u;
}

// ---- split-K tiles reduced by the consumer ----
// The tensor-core GEMM splits its (feature tile, token tile, K block) units
// into one contiguous stream-K range per CTA: CTA i owns units
// [range_start(i), range_start(i + 1)).  A tile whose units all fall in one
// CTA is written whole by that CTA.  In deferred mode a tile split over CTAs
// i0..i1 is not reduced by the GEMM: each CTA stores its fp32 partial in the
// workspace slot (i, s) -- s = 0 if the tile is the first of i's range, else
// 1 -- as [BN rows][128 features], and leaves Y untouched.  The kernel that
// next reads Y (RMSNorm, RoPE) forms the value itself: Y (accumulate) or the
// bias (store), plus the sum of the partials in CTA order, which keeps the
// result deterministic and takes the reduction off the GEMM's tail.
__host__ __device__ inline long long range_start(long long i, long long total, int grid) {
  return i * total / grid;
}
// CTA whose range holds unit u
__host__ __device__ inline int cta_of(long long u, long long total, int grid) {
  return (int)(((u + 1) * grid - 1) / total);
}

struct SplitView {
  const float *ws = nullptr;    // null: Y is complete
  const float *bias = nullptr;  // store mode: added to split tiles
  long long total = 0;
  int grid = 0, KB = 0, BN = 0, m_tiles = 0;
  int accum = 0;  // 1: Y holds the old value the product adds to
  int small = 0;  // 1: (total + 1) * grid < 2^31, so 32-bit index math is exact
};

// CTAs i0..i1 hold the units of tile tl; the tile is i0's slot s0 and the
// slot 0 of every later CTA (their ranges start inside it).
struct SplitTile {
  int i0, i1, s0;
};
__device__ __forceinline__ SplitTile split_tile(const SplitView &sv, long long tl) {
  SplitTile st;
  if (sv.small) {
    const unsigned u0 = (unsigned)tl * (unsigned)sv.KB, T = (unsigned)sv.total,
                   g = (unsigned)sv.grid;
    st.i0 = (int)(((u0 + 1) * g - 1) / T);
    st.i1 = (int)(((u0 + sv.KB) * g - 1) / T);
    st.s0 = (unsigned)st.i0 * T / g >= u0 ? 0 : 1;
    return st;
  }
  const long long u0 = tl * sv.KB;
  st.i0 = cta_of(u0, sv.total, sv.grid);
  st.i1 = cta_of(u0 + sv.KB - 1, sv.total, sv.grid);
  st.s0 = range_start(st.i0, sv.total, sv.grid) >= u0 ? 0 : 1;
  return st;
}

// Sum of the partials of split tile st at element offset `off` within a slot
// ([BN][128] fp32), in CTA order.  A deferred GEMM splits no tile over more
// than SPLIT_MAX_PARTS CTAs, so the code is straight-line: every load is
// issued before the first add and the sum costs one round trip to L2.
constexpr int SPLIT_MAX_PARTS = 8;
__device__ __forceinline__ float4 split_sum4(const SplitView &sv, const SplitTile &st, size_t off) {
  const size_t slot = (size_t)sv.BN * 128;
  float4 x[SPLIT_MAX_PARTS];
  x[0] = __ldcg((const float4 *)(sv.ws + ((size_t)st.i0 * 2 + st.s0) * slot + off));
#pragma unroll
  for (int j = 1; j < SPLIT_MAX_PARTS; ++j)
    if (st.i0 + j <= st.i1) x[j] = __ldcg((const float4 *)(sv.ws + (size_t)(st.i0 + j) * 2 * slot + off));
  float4 acc = x[0];
#pragma unroll
  for (int j = 1; j < SPLIT_MAX_PARTS; ++j)
    if (st.i0 + j <= st.i1) {
      acc.x += x[j].x;
      acc.y += x[j].y;
      acc.z += x[j].z;
      acc.w += x[j].w;
    }
  return acc;
}
__device__ __forceinline__ float split_sum(const SplitView &sv, const SplitTile &st, size_t off) {
  const size_t slot = (size_t)sv.BN * 128;
  float x[SPLIT_MAX_PARTS];
  x[0] = __ldcg(sv.ws + ((size_t)st.i0 * 2 + st.s0) * slot + off);
#pragma unroll
  for (int j = 1; j < SPLIT_MAX_PARTS; ++j)
    if (st.i0 + j <= st.i1) x[j] = __ldcg(sv.ws + (size_t)(st.i0 + j) * 2 * slot + off);
  float acc = x[0];
#pragma unroll
  for (int j = 1; j < SPLIT_MAX_PARTS; ++j)
    if (st.i0 + j <= st.i1) acc += x[j];
  return acc;
}

// Value of Y[t][n..n+3] (n % 4 == 0, one tile) given the raw Y entries y.
__device__ __forceinline__ float4 split_value4(const SplitView &sv, const SplitTile &st, float4 y,
                                               int t, int n) {
  if (!sv.ws || st.i0 == st.i1) return y;
  const int mt = t / sv.BN;
  const float4 acc = split_sum4(sv, st, (size_t)(t - mt * sv.BN) * 128 + (n & 127));
  float4 b = y;
  if (!sv.accum) b = sv.bias ? *(const float4 *)(sv.bias + n) : make_float4(0.f, 0.f, 0.f, 0.f);
  return make_float4(b.x + acc.x, b.y + acc.y, b.z + acc.z, b.w + acc.w);
}
__device__ __forceinline__ float split_value(const SplitView &sv, const SplitTile &st, float y,
                                             int t, int n) {
  if (!sv.ws || st.i0 == st.i1) return y;
  const int mt = t / sv.BN;
  const float acc = split_sum(sv, st, (size_t)(t - mt * sv.BN) * 128 + (n & 127));
  return (sv.accum ? y : (sv.bias ? sv.bias[n] : 0.f)) + acc;
}

struct TcWorkspace {
  float *partials;  // gemm_tc_ws_bytes(num_sms)
  int *counters;    // 2 * max_tiles zeroed ints (arrivals, published parts)
  int *dev_flag;
  int num_sms;
  long long max_tiles;
};

// Accumulated device time of one kernel class.
struct ProfClass {
  std::string name;
  double ms = 0;
  int64_t launches = 0;
  int64_t bytes = 0;
};

}  // namespace kvr

struct kvr_cache;

struct kvr_model {
  kvr::Dims dims{};
  std::vector<kvr_cache *> caches;  // live caches, freed with the model
  void *weight_block = nullptr;
  size_t weight_bytes = 0;
  void *embed = nullptr, *lm_head = nullptr;
  float *final_norm = nullptr;
  std::vector<kvr::LayerW> layers;
  float2 *rope = nullptr;  // [max_ctx + reserve][dh/2] (cos, sin), fp32 from fp64 angles
  CUtensorMap tm_lm;
  bool tc_lm = false;
  kvr::TcWorkspace tcw{};
  int4 *blocks_d = nullptr;      // attention query blocks of the current pass
  int max_blocks = 0;
  float *attn_ws_o = nullptr;    // split-KV partials
  float2 *attn_ws_ml = nullptr;
  size_t attn_ws_floats = 0;
  bool use_tc = true;  // tensor-core GEMM for bf16 shapes it takes
  bool use_graphs = true;  // CUDA graphs for repeated repair passes
  cudaStream_t stream = nullptr;
  int device = 0;
  int num_sms = 0;
  // workspace
  void *ws_block = nullptr;
  int32_t *pos_d = nullptr;  // [R] positions of the rows of a pass
  int32_t *rowdoc_d = nullptr;  // [R] batch: document of each row
  float *h = nullptr, *qkv = nullptr, *q = nullptr, *gu = nullptr, *logits = nullptr;
  void *qb = nullptr;  // bf16 post-RoPE q for the tensor-core attention
  void *a = nullptr, *attn = nullptr, *act = nullptr;
  float *scores = nullptr;     // [max_ctx + reserve] selector scores
  unsigned long long *keys = nullptr;  // [max_ctx + reserve] top-K keys
  int32_t *sel_out = nullptr;  // [max_ctx] selected positions
  int32_t *sel_count = nullptr;
  void *read_scratch = nullptr;  // cache readback: positions, then the gathered K and V
  size_t read_scratch_bytes = 0;
  // kvr_repair_read: the pass's K/V rows as RoPE writes them, copied to the
  // host group by group (on rd_stream, after the graph's rd_ev[g]) while the
  // pass goes on; rd_cap carries the events' side branch inside a capture
  void *rows_scratch = nullptr;
  size_t rows_scratch_bytes = 0;
  cudaStream_t rd_stream = nullptr, rd_cap = nullptr;
  cudaEvent_t rd_ev[kvr::KVR_RD_GROUPS] = {}, rd_fork[kvr::KVR_RD_GROUPS] = {};
  cudaEvent_t rd_join = nullptr;
  void *sel_scratch = nullptr;   // selector: edited tokens, saved stale rows, probabilities
  size_t sel_scratch_bytes = 0;
  void *batch_scratch = nullptr; // batched repair: documents' TMA views, cache views, tokens
  size_t batch_scratch_bytes = 0;
  int *dev_flag = nullptr;     // device error flag (bounded waits)
  kvr::TraceBuf trace{};       // attached device timeline buffer, if any
  kvr::SplitView pending{};    // split tiles of h not yet added (next RMSNorm adds them)
  bool defer_splits = true;    // GEMM split tiles reduced by the consumer
  bool use_tc5 = true;         // tcgen05 attention for single-document passes
  bool use_chain = false;      // a pass's projections and norms as GEMM chains (opt-in)
  unsigned *chain_bar = nullptr;  // hand-off counters of a pass's chains, zeroed per pass
  // pinned staging for host->device argument copies
  int32_t *stage_h = nullptr;
  int32_t *stage_d = nullptr;
  size_t stage_cap = 0;
  size_t stage_off = 0;           // next free slot (copies take consecutive slots)
  cudaEvent_t stage_ev = nullptr;  // recorded after the last staged copy
  int32_t *rb_h = nullptr;         // pinned readback: selector count, flag, positions
  int32_t *flag_h = nullptr;       // pinned readback of the device error flag
  // profiling
  bool prof = false;
  std::vector<kvr::ProfClass> prof_classes;
  std::vector<std::pair<int, std::pair<cudaEvent_t, cudaEvent_t>>> prof_pending;
  int64_t launches = 0;
};

struct kvr_cache {
  kvr_model *model = nullptr;
  int n = 0, cap = 0, n_pages = 0;
  void *pages = nullptr;
  int32_t *table = nullptr;   // device [n_pages]
  // TMA view of the page pool (bf16): rows of head_dim elements, one row per
  // (page, layer, k|v, kv head, slot); boxes of 64 rows x 64 elements
  CUtensorMap tm_kv{};
  bool tm_kv_ok = false;
  int32_t *tokens_d = nullptr;  // device [cap]
  std::vector<int32_t> tokens_h;
  bool poisoned = false;
  struct Graph {
    int M, nb, ns;
    const void *rows_out;  // kvr_repair_read's row buffer, or null
    int64_t kernels;
    cudaGraphExec_t exec;
  };
  std::vector<Graph> graphs;  // captured repair passes of this cache
  kvr::KVView view() const {
    return kvr::KVView{pages, table, model->dims.L, model->dims.G, model->dims.dh};
  }
};

namespace kvr {

// ---- device timeline trace ----
// With a buffer attached, thread 0 of every CTA of the pass kernels appends
// one record of 16 words: kind | smid << 8 | linear block index << 16; the
// time the CTA started; the time its wait on the predecessor kernel returned;
// the time it finished; eight kernel-specific marks (0 where unset); four
// zero words (%globaltimer, ns).  GEMM marks, each for the CTA's last tile:
// 0 first operand stage landed, 1 all MMAs complete, 2 accumulator taken by
// the epilogue, 3 partial tile stored, 4 split-tile arrival counted
// (stream-K) or partials staged across the cluster, 5 tile reduced and
// written, 6 epilogue warps done, 7 all warps done.  Attention mark: 0 last key
// chunk consumed.  The buffer pointer lives in constant memory (one copy per
// translation unit, set by its trace_attach_* function).  Even detached, the
// checks lengthen each kernel's critical path, so tracing is compiled only
// into the KVR_TRACE build of the library; elsewhere the hooks are empty.
enum TraceKind : int {
  TK_EMBED = 1, TK_NORM, TK_GEMM, TK_ROPE, TK_ATTN, TK_COMBINE, TK_OTHER, TK_SELECT, TK_SELECT_ACC
};
#ifdef KVR_TRACE
static __constant__ TraceBuf g_trace;

__device__ __forceinline__ unsigned long long trace_now() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Stamps of thread 0's CTA, in shared memory: start, wait, marks 0..7.
__device__ __forceinline__ unsigned long long *trace_stamps() {
  __shared__ unsigned long long t[10];
  return t;
}

// Kernel-specific mark i (0..7), by any one thread of the CTA.
__device__ __forceinline__ void trace_mark(int i) {
  if (g_trace.rec) trace_stamps()[2 + i] = trace_now();
}

struct TraceScope {
  int kind;
  __device__ explicit TraceScope(int k) : kind(k) {
    if (threadIdx.x == 0 && g_trace.rec) {
      unsigned long long *t = trace_stamps();
      t[0] = t[1] = trace_now();
#pragma unroll
      for (int i = 2; i < 10; ++i) t[i] = 0;
    }
  }
  __device__ void waited() {
    if (threadIdx.x == 0 && g_trace.rec) trace_stamps()[1] = trace_now();
  }
  __device__ void finish() {
    if (threadIdx.x != 0 || !g_trace.rec) return;
    unsigned long long *t = trace_stamps();
    if (t[0] == 0) return;
    unsigned long long t2 = trace_now();
    unsigned int i = atomicAdd(g_trace.count, 1u);
    if (i < g_trace.cap) {
      unsigned int smid;
      asm volatile("mov.u32 %0, %%smid;" : "=r"(smid));
      unsigned long long blk =
          blockIdx.x +
          (unsigned long long)gridDim.x * (blockIdx.y + (unsigned long long)gridDim.y * blockIdx.z);
      unsigned long long *r = g_trace.rec + 16ull * i;
      r[0] = (unsigned long long)kind | (unsigned long long)(smid & 0xff) << 8 | blk << 16;
      r[1] = t[0];
      r[2] = t[1];
      r[3] = t2;
#pragma unroll
      for (int k = 0; k < 8; ++k) r[4 + k] = t[2 + k];
#pragma unroll
      for (int k = 12; k < 16; ++k) r[k] = 0;
    }
    t[0] = 0;
  }
  __device__ ~TraceScope() { finish(); }
};
#else
__device__ __forceinline__ void trace_mark(int) {}
struct TraceScope {
  __device__ explicit TraceScope(int) {}
  __device__ void waited() {}
  __device__ void finish() {}
};
#endif

#ifdef KVR_TRACE
#define KVR_TRACE_ATTACH(fn)                                           \
  cudaError_t fn(const kvr::TraceBuf &b) {                             \
    return cudaMemcpyToSymbol(kvr::g_trace, &b, sizeof(kvr::TraceBuf)); \
  }
#else
#define KVR_TRACE_ATTACH(fn) \
  cudaError_t fn(const kvr::TraceBuf &) { return cudaSuccess; }
#endif
cudaError_t trace_attach_rows(const TraceBuf &b);
cudaError_t trace_attach_gemm(const TraceBuf &b);
cudaError_t trace_attach_attn(const TraceBuf &b);
cudaError_t trace_attach_attn5(const TraceBuf &b);
cudaError_t trace_attach_select(const TraceBuf &b);

// ---- programmatic dependent launch (PDL) ----
// Kernels of a pass are launched with programmatic stream serialisation: a
// kernel may start while its predecessor drains.  Every such kernel calls
// pdl_trigger() on entry (its own successor may then be scheduled) and
// pdl_wait() before it touches anything its predecessors write; pdl_wait()
// returns once the predecessor grid has completed and its memory is visible.
// Without the launch attribute both are no-ops.
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

extern bool g_pdl;  // launch with the PDL attribute (KVR_DISABLE_PDL=1 turns it off)

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g_pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Message returned by kvr_last_error() on the calling thread.
void set_last_error(const char *msg);

// ---- allocation (allocator hook) ----
void *dev_alloc(size_t bytes);
void dev_free(void *p);

// ---- kernels: weights ----
// Fill rows of a device tensor from the seeded generator.  Element (r, c) of
// the canonical [rows][cols] tensor is generated and stored at
// dst[map(r) * cols + c] with map(r) = row_off + r (interleave == 0) or the
// gate/up interleave (interleave == 1: gate, 2: up).  out_f32: store as fp32
// (value first rounded to the model dtype).
void launch_init_tensor(void *dst, int dtype, bool out_f32, uint64_t tensor_seed, double scale,
                        int64_t rows, int64_t cols, int64_t row_off, int interleave,
                        cudaStream_t s);
void launch_fill_f32(float *dst, float v, size_t n, cudaStream_t s);

// ---- kernels: row ops ----
void launch_embed_rows(const void *embed, int dtype, const int32_t *tokens,
                       const int32_t *const *doc_tokens, const int32_t *rowdoc,
                       const int32_t *pos, int M, int d, float *h, cudaStream_t s);
// Rows row0 .. row0+M-1 of h; out row i is h row row0 + i.  With a split
// view (rows indexed from h's base), the completed rows are written back to h.
void launch_rmsnorm(float *h, const float *g, int row0, int M, int d, double eps, void *out,
                    int out_dtype, cudaStream_t s, const SplitView *sv = nullptr);
// q_out: fp32 rotated q; qb_out (optional): bf16 rotated q times qscale;
// rows_out (optional, with write_kv): the K/V rows as written into the cache,
// K then V, each [M][L][G][dh] in the cache dtype.
void launch_rope_scatter(const float *qkv, const float2 *rope, const int32_t *pos, int M,
                         const Dims &dm, int layer, const KVView *views, const int32_t *rowdoc,
                         KVView single, float *q_out, void *qb_out, float qscale, bool write_kv,
                         cudaStream_t s, const SplitView *sv = nullptr, void *rows_out = nullptr);
void launch_swiglu(const float *gu, int M, int F, void *act, int dtype, cudaStream_t s);
void launch_cache_gather(KVView v, int dtype, const int32_t *pos, int n_pos, int l0, int l1,
                         int G, int dh, float *k_out, float *v_out, cudaStream_t s);
// The same gather in the cache's element type (no widening).
void launch_cache_gather_raw(KVView v, int dtype, const int32_t *pos, int n_pos, int l0, int l1,
                             int G, int dh, void *k_out, void *v_out, cudaStream_t s);
// Rows [n_pos][L][G][dh] (cache dtype) of consecutive positions p0.. into the pages.
void launch_cache_scatter_raw(KVView v, int dtype, int p0, int n_pos, const void *k_in,
                              const void *v_in, cudaStream_t s);
void launch_rows_copy(KVView v, int dtype, const int32_t *pos, int n_pos, int l0, int l1,
                      void *buf, bool to_buf, cudaStream_t s);
void launch_transplant(KVView dst, KVView src, int dtype, const int32_t *pos, int n_pos,
                       cudaStream_t s);
void launch_row_logprob(const float *logits, int rows, int V, const int32_t *target, float *out,
                        cudaStream_t s);

// ---- kernels: GEMM  Y[M][N] (+)= X[M][K] W[N][K]^T (+ bias) ----
struct GemmArgs {
  const void *X;
  const void *W;
  const float *bias;
  float *Y;
  int M, N, K;
  int ldx, ldy;
  int dtype;       // operands: KVR_DTYPE_F32 or KVR_DTYPE_BF16
  int accumulate;  // 1: Y += result
};
void launch_gemm_simt(const GemmArgs &g, cudaStream_t s);

// Tensor-core GEMM (bf16, N % 128 == 0, K % 64 == 0).  Epilogues:
enum { GEMM_EPI_STORE = 0, GEMM_EPI_ACCUM = 1, GEMM_EPI_SWIGLU = 2 };
bool make_tmap_bf16(CUtensorMap *map, const void *ptr, int rows, int cols, int box_rows);
// Weights of the tensor-core GEMM are stored blocked: the 128-row x 64-column
// tile (feature tile nt, K block kb) of W [N][K] is one contiguous 16 KB
// block, row-major inside, block nt * K/64 + kb -- so each TMA box the GEMM
// loads is one run of DRAM.  make_tmap_weight: the tensor map of such a
// weight (rows of 64 elements); launch_weight_tile: row-major <-> blocked
// (untile), between distinct buffers of N*K bf16.
bool make_tmap_weight(CUtensorMap *map, const void *w, int N, int K);
const char *launch_weight_tile(const void *src, void *dst, int N, int K, bool untile,
                               cudaStream_t s);
bool gemm_tc_supported(int N, int K);
int gemm_tc_bn(int M);
size_t gemm_tc_ws_bytes(int num_sms);
// GEMM_EPI_SWIGLU: W rows interleaved gate/up in blocks of 16; writes
// out2[t][f] = bf16(silu(gate) * up), f < N/2, row stride ld2.
// Returns nullptr on success, else what went wrong.
// defer: leave split tiles to the consumer and describe them in *defer
// (ws stays null when no tile was split, or when a tile would span more
// than SPLIT_MAX_PARTS CTAs: then the GEMM reduces them itself).  Not for
// the SwiGLU epilogue, which needs complete sums.
// One step of a GEMM chain (launch_gemm_chain): a tensor-core GEMM with
// launch_gemm_tc's arguments, or an RMSNorm of the chain's rows (h completed
// in place from the previous GEMM's deferred split tiles, out in bf16).
struct ChainStep {
  bool norm = false;
  GemmArgs g{};
  const CUtensorMap *tmW = nullptr;
  int epi = 0;
  void *out2 = nullptr;
  int ld2 = 0;
  bool defer = false;  // split tiles left to the next step (a norm) or kernel
  float *h = nullptr;
  const float *gain = nullptr;
  float eps = 0.f;
  int d = 0;
  void *out = nullptr;
};
// Up to 6 steps (at most 4 GEMMs, 2 norms) in one persistent launch of
// num_sms CTAs; every GEMM has the same rows M (<= num_sms when a norm is
// present) and at least num_sms stream-K units.  bar: gemm_chain_bar_words()
// zeroed device words for this launch.  last_defer: the last GEMM's deferred
// split tiles (ws null when it has none).  nullptr on success.
size_t gemm_chain_bar_words();
const char *launch_gemm_chain(const ChainStep *steps, int n, const TcWorkspace &ws, unsigned *bar,
                              cudaStream_t s, SplitView *last_defer);
const char *launch_gemm_tc(const GemmArgs &g, const CUtensorMap &tmW, int epi, void *out2,
                           int ld2, const TcWorkspace &ws, cudaStream_t s,
                           SplitView *defer = nullptr);

// ---- kernels: attention ----
// o[i] = softmax(q_i K[0..pos_i]^T / sqrt(dh)) V[0..pos_i] for every row i,
// GQA head h -> kv head h / (H/G).  q fp32 [M][H*dh]; out [M][H*dh] in dtype.
void launch_attention_simt(const float *q, const int32_t *pos, int M, const Dims &dm, int layer,
                           const KVView *views, const int32_t *rowdoc, KVView single, void *out,
                           cudaStream_t s);

// Tensor-core attention (bf16 cache, head_dim 64 or 128).  blocks: device
// int4 (row0, nrows, kmax, doc) per query block (rows of one document, at
// most attn_tc_rows_per_block(grp) rows, kmax = largest position); the
// keys 0..kmax of each block are split into n_splits ranges of 64-key
// chunks (ws_o/ws_ml hold the partials when n_splits > 1).
int attn_tc_rows_per_block(int grp);
size_t attn_tc_ws_floats(int n_splits, int n_blocks, int G, int dh);
// q: bf16 [M][H*dh], rotated (the kernels scale the scores by log2(e)/sqrt(dh)).
const char *launch_attention_tc(const void *q, const int32_t *pos, const int4 *blocks,
                                int n_blocks, int max_rows_per_block, int n_splits, const Dims &dm,
                                int layer, const KVView *views, KVView single, float *ws_o,
                                float2 *ws_ml, void *out, cudaStream_t s);
// The split merge alone (after launch_attention_tc5 with n_splits > 1).
// prefetch (optional): the next GEMM's weights, pulled into L2 while the
// combine (bound by L2 latency, not HBM) runs.
const char *launch_attention_combine(const int4 *blocks, int n_blocks, int max_rows_per_block,
                                     int n_splits, const Dims &dm, float *ws_o, float2 *ws_ml,
                                     void *out, cudaStream_t s, const void *prefetch = nullptr,
                                     long long prefetch_bytes = 0);
// tcgen05 attention (bf16 cache, head_dim 64 or 128): query blocks of at most
// attn_tc5_rows_per_block(grp) rows of one document each; partials in the
// same workspace layout as launch_attention_tc.  One document: pages, table
// and tm_kv (its TMA view).  Several: views and tmaps, device arrays indexed
// by a block's document (blocks[].w), tmaps 64-byte aligned.
int attn_tc5_rows_per_block(int grp);
int attn_tc5_ctas_per_sm(int dh);
const char *launch_attention_tc5(const void *q, const int32_t *pos, const int4 *blocks,
                                 int n_blocks, int n_splits, const Dims &dm, int layer,
                                 const void *pages, const int32_t *table, const CUtensorMap &tm_kv,
                                 float *ws_o, float2 *ws_ml, void *out, int *dev_flag,
                                 cudaStream_t s, const KVView *views = nullptr,
                                 const CUtensorMap *tmaps = nullptr);

// ---- kernels: selectors ----
// The keys of a simple policy (EditLocal, Structural, Random,
// EditLocal@boundary), generated inside the top-K kernel instead of read from
// a keys array.
struct SimpleKeys {
  int policy = -1;                  // < 0: the top-K reads the keys array
  const int32_t *tokens = nullptr;  // the edited context (device)
  int delim = 0;
  uint64_t seed = 0;
  const int *bound = nullptr;       // EditLocal@boundary: launch_first_delim's result
};
// EditLocal@boundary: the first delimiter position at or after s_end into
// *bound, which must hold n - 1 on entry.
void launch_first_delim(const int32_t *tokens, int n, int s_end, int delim, int *bound,
                        cudaStream_t s);
// Attention selector, one layer: adds to scores[j], j in [s_end, n), the
// pool-softmax probabilities of the S span rows' queries (fp32 q, [S][H*dh]).
// ws_base: attn_select_ws_bytes(S, dm, n - s_end) bytes; first_layer zeroes
// its arrival counts.
size_t attn_select_ws_bytes(int S, const Dims &dm, int n_pool);
void launch_attn_select_scores(const float *q, int S, const Dims &dm, int layer, KVView v,
                               int s_end, int n, void *ws_base, bool first_layer,
                               float *scores, cudaStream_t s);
void launch_kv_deviation(const float *qkv, const float2 *rope, const int32_t *pos, int M,
                         const Dims &dm, KVView v, float *scores, cudaStream_t s);
void launch_float_keys(const float *scores, int n, int s_end, unsigned long long *keys,
                       cudaStream_t s);
// flag_in (optional): the device error flag, copied to *flag_out once every
// kernel queued before has run, so that one readback returns both.
const char *launch_topk(const unsigned long long *keys, int n, int s_end, int K, int32_t *out,
                        int32_t *count, cudaStream_t s, const SimpleKeys &gen = SimpleKeys{},
                        const int *flag_in = nullptr, int32_t *flag_out = nullptr);

}  // namespace kvr
