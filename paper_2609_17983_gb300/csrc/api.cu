// api.cu -- the C ABI of libkvrepair and its host-side orchestration.
//
// Every entry point validates its arguments on the host, then enqueues the
// layer-major pass of the repair operator R (Sec. 3, Eq. 1) on the model's
// stream: embedding gather of the rows, then per layer RMSNorm -> QKV GEMM ->
// RoPE at the original positions + K/V scatter of all rows -> scattered-query
// attention -> O GEMM (+residual) -> RMSNorm -> gate/up GEMM -> SwiGLU ->
// down GEMM (+residual).
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "kvr_internal.cuh"

using namespace kvr;

namespace {

thread_local std::string g_err;

kvr_status fail(kvr_status code, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

kvr_alloc_fn g_alloc = nullptr;
kvr_free_fn g_free = nullptr;
void *g_alloc_ctx = nullptr;

#define CUDA_TRY(expr)                                                                   \
  do {                                                                                   \
    cudaError_t e__ = (expr);                                                            \
    if (e__ != cudaSuccess)                                                              \
      return fail(e__ == cudaErrorMemoryAllocation ? KVR_E_NOMEM : KVR_E_CUDA, "%s: %s", \
                  #expr, cudaGetErrorString(e__));                                       \
  } while (0)

#define KVR_TRY(expr)           \
  do {                          \
    kvr_status s__ = (expr);    \
    if (s__ != KVR_OK) return s__; \
  } while (0)

kvr_status launch_check(kvr_model *m, int kernels) {
  m->launches += kernels;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(KVR_E_CUDA, "kernel launch: %s", cudaGetErrorString(e));
  return KVR_OK;
}

// ------------------------------------------------------------ profiling

enum ProfId {
  P_EMBED, P_NORM, P_GEMM_QKV, P_ROPE, P_ATTN, P_GEMM_O, P_GEMM_GU, P_SWIGLU, P_GEMM_DOWN,
  P_LMHEAD, P_SELECT, P_GEMM_CHAIN, P_NCLASS
};
const char *kProfNames[P_NCLASS] = {"embed",  "rmsnorm",  "gemm_qkv",  "rope_scatter",
                                    "attention", "gemm_o", "gemm_gu",   "swiglu",
                                    "gemm_down", "lm_head", "select",    "gemm_chain"};

struct Prof {
  kvr_model *m;
  int cls;
  int64_t bytes;
  cudaEvent_t a = nullptr, b = nullptr;
  Prof(kvr_model *mm, int c, int64_t by) : m(mm), cls(c), bytes(by) {
    if (!m->prof) return;
    cudaEventCreate(&a);
    cudaEventCreate(&b);
    cudaEventRecord(a, m->stream);
  }
  ~Prof() {
    if (!m->prof || !a) return;
    cudaEventRecord(b, m->stream);
    m->prof_pending.push_back({cls, {a, b}});
    m->prof_classes[cls].launches += 1;
    m->prof_classes[cls].bytes += bytes;
  }
};

void prof_collect(kvr_model *m) {
  for (auto &p : m->prof_pending) {
    float ms = 0.f;
    cudaEventSynchronize(p.second.second);
    cudaEventElapsedTime(&ms, p.second.first, p.second.second);
    m->prof_classes[p.first].ms += ms;
    cudaEventDestroy(p.second.first);
    cudaEventDestroy(p.second.second);
  }
  m->prof_pending.clear();
}

// ------------------------------------------------------------ staging

// Copy host int32 data to device through the model's pinned staging buffer.
// Copies take consecutive 128-byte-aligned slots, so a call does not wait for
// the copies queued before it; when the next slot would not fit, the buffer
// starts over after every queued copy has completed.
kvr_status stage_h2d(kvr_model *m, int32_t *dst_dev, const int32_t *src, size_t count) {
  if (count == 0) return KVR_OK;
  if (count > m->stage_cap) return fail(KVR_E_UNSUPPORTED, "staging overflow (%zu)", count);
  if (m->stage_off + count > m->stage_cap) {
    CUDA_TRY(cudaEventSynchronize(m->stage_ev));
    m->stage_off = 0;
  }
  int32_t *h = m->stage_h + m->stage_off;
  memcpy(h, src, count * sizeof(int32_t));
  CUDA_TRY(cudaMemcpyAsync(dst_dev, h, count * sizeof(int32_t), cudaMemcpyHostToDevice,
                           m->stream));
  CUDA_TRY(cudaEventRecord(m->stage_ev, m->stream));
  m->stage_off += (count + 31) / 32 * 32;
  return KVR_OK;
}

// ------------------------------------------------------------ GEMM dispatch

// Y (+)= X W^T through the tensor-core kernel when the weight has a TMA
// descriptor, else the FFMA kernel.  epi selects the epilogue; for SwiGLU
// the FFMA path writes gate/up to m->gu and runs the SwiGLU kernel.
// defer: split tiles of the tensor-core GEMM are left to the kernel that
// next reads Y, which must take *defer (ws null when Y is complete).
kvr_status gemm(kvr_model *m, int cls, const void *X, const void *W, const CUtensorMap *tm,
                const float *bias, float *Y, int M, int N, int K, int epi,
                SplitView *defer = nullptr) {
  const Dims &dm = m->dims;
  Prof pr(m, cls, (int64_t)N * K * (int64_t)dm.es());
  if (defer) *defer = SplitView{};
  if (tm && m->use_tc) {
    GemmArgs g{X, W, bias, Y, M, N, K, K, N, dm.dtype, epi == GEMM_EPI_ACCUM};
    const char *e = launch_gemm_tc(g, *tm, epi, epi == GEMM_EPI_SWIGLU ? m->act : nullptr,
                                   N / 2, m->tcw, m->stream, m->defer_splits ? defer : nullptr);
    if (e) return fail(KVR_E_CUDA, "tensor-core GEMM (M=%d N=%d K=%d): %s", M, N, K, e);
    return launch_check(m, 1);
  }
  if (epi == GEMM_EPI_SWIGLU) {
    GemmArgs g{X, W, nullptr, m->gu, M, N, K, K, N, dm.dtype, 0};
    launch_gemm_simt(g, m->stream);
    launch_swiglu(m->gu, M, N / 2, m->act, dm.dtype, m->stream);
    return launch_check(m, 2);
  }
  GemmArgs g{X, W, bias, Y, M, N, K, K, N, dm.dtype, epi == GEMM_EPI_ACCUM};
  launch_gemm_simt(g, m->stream);
  return launch_check(m, 1);
}

// ------------------------------------------------------------ the pass

struct Rows {
  int M = 0;
  const int32_t *pos = nullptr;              // device [M]
  const int32_t *tokens = nullptr;           // device tokens of a single document
  const int32_t *const *doc_tokens = nullptr;  // device [docs] (batch)
  const int32_t *rowdoc = nullptr;           // device [M] (batch)
  const KVView *views = nullptr;             // device [docs] (batch)
  KVView single{};
  int max_pos = 0;                           // largest position among the rows
  const int4 *blocks = nullptr;              // attention query blocks (device)
  int n_blocks = 0, n_splits = 1, max_block_rows = 0;
  const CUtensorMap *tm_kv = nullptr;        // TMA view of the single document's pages
  const CUtensorMap *tmaps = nullptr;        // device [docs]: TMA views of a batch's pages
  bool tc5 = false;                          // attention on tcgen05 (set by plan_attention)
  // kvr_repair_read: RoPE also writes the rows' K/V to rows_out (K then V,
  // [M][L][G][dh]); after every rd_every layers an event marks them ready
  void *rows_out = nullptr;
  int rd_every = 0;
};

bool use_tc_attention(const kvr_model *m) {
  return m->dims.dtype == KVR_DTYPE_BF16 && (m->dims.dh == 64 || m->dims.dh == 128);
}

// Query blocks for the tensor-core attention: consecutive rows of one
// document (rows of a document are in ascending position order), at most
// rows_per_block rows; and a key split count giving about two CTAs per SM.
kvr_status plan_attention(kvr_model *m, Rows &r, const int32_t *pos, const int32_t *rowdoc) {
  r.tc5 = false;
  if (!use_tc_attention(m) || r.M <= 0) return KVR_OK;
  const Dims &dm = m->dims;
  const int grp = dm.H / dm.G;
  // the tcgen05 kernel (query blocks of up to 128 query vectors) when every
  // document has a TMA view of its pages, else the mma.sync kernel
  r.tc5 = m->use_tc5 && (rowdoc ? r.tmaps != nullptr : r.tm_kv != nullptr) &&
          attn_tc5_rows_per_block(grp) > 0;
  const int qb = r.tc5 ? attn_tc5_rows_per_block(grp) : attn_tc_rows_per_block(grp);
  std::vector<int32_t> b;
  int max_chunks = 0, max_rows = 0;
  for (int i = 0; i < r.M;) {
    int doc = rowdoc ? rowdoc[i] : 0;
    int e = i;
    while (e < r.M && (rowdoc ? rowdoc[e] : 0) == doc) ++e;
    // the document's rows in equal blocks of at most qb rows
    const int nbd = (e - i + qb - 1) / qb, per = (e - i + nbd - 1) / nbd;
    for (int j0 = i; j0 < e; j0 += per) {
      const int j1 = std::min(e, j0 + per);
      const int kmax = pos[j1 - 1];
      max_rows = std::max(max_rows, j1 - j0);
      b.insert(b.end(), {j0, j1 - j0, kmax, doc});
      max_chunks = std::max(max_chunks, kmax / KVR_PAGE + 1);
    }
    i = e;
  }
  int nb = (int)b.size() / 4;
  if (nb > m->max_blocks) return fail(KVR_E_UNSUPPORTED, "too many attention blocks (%d)", nb);
  // about one wave: as many CTAs as fit on the SMs at once
  const int target = m->num_sms * (r.tc5 ? attn_tc5_ctas_per_sm(dm.dh) : 1);
  int splits = r.tc5 ? std::max(1, target / (nb * dm.G))  // one wave: no straggler CTAs
                     : std::max(1, (target + nb * dm.G - 1) / (nb * dm.G));
  splits = std::min(std::min(splits, max_chunks), 64);  // the combine merges <= 64 splits
  while (splits > 1 && attn_tc_ws_floats(splits, nb, dm.G, dm.dh) > m->attn_ws_floats) --splits;
  KVR_TRY(stage_h2d(m, (int32_t *)m->blocks_d, b.data(), b.size()));
  r.blocks = m->blocks_d;
  r.n_blocks = nb;
  r.n_splits = splits;
  r.max_block_rows = max_rows;
  return KVR_OK;
}

kvr_status embed(kvr_model *m, const Rows &r) {
  Prof pr(m, P_EMBED, (int64_t)r.M * m->dims.d * (int64_t)m->dims.es());
  m->pending = SplitView{};
  launch_embed_rows(m->embed, m->dims.dtype, r.tokens, r.doc_tokens, r.rowdoc, r.pos, r.M,
                    m->dims.d, m->h, m->stream);
  return launch_check(m, 1);
}

// RMSNorm of h rows row0 .. row0+M-1 into m->a, first adding the split
// tiles a deferred GEMM left pending in h.
kvr_status norm(kvr_model *m, const float *g, int M, int row0 = 0) {
  Prof pr(m, P_NORM, (int64_t)M * m->dims.d * 4);
  launch_rmsnorm(m->h, g, row0, M, m->dims.d, m->dims.eps, m->a, m->dims.dtype, m->stream,
                 &m->pending);
  m->pending = SplitView{};
  return launch_check(m, 1);
}

// QKV projection, RoPE, and (write_kv) the K/V scatter of layer l.  keep_qkv:
// m->qkv must hold the complete projection afterwards (else split tiles of
// the GEMM are completed by the RoPE kernel alone).  need_q: the fp32 q
// (m->q) is read afterwards (attention selector); the tensor-core attention
// reads only the bf16 q, and the fp32 one is then not written.
// RoPE of layer l's projection in m->qkv (completed from sv, the QKV GEMM's
// deferred split tiles), q to m->qb (and m->q when need_q or no tensor-core
// attention), and (write_kv) the K/V rows into the cache.
kvr_status rope(kvr_model *m, const Rows &r, int l, bool write_kv, bool need_q,
                const SplitView &sv) {
  const Dims &dm = m->dims;
  Prof pr(m, P_ROPE, (int64_t)r.M * dm.Nqkv() * 4);
  const bool tc = use_tc_attention(m);
  launch_rope_scatter(m->qkv, m->rope, r.pos, r.M, dm, l, r.views, r.rowdoc, r.single,
                      tc && !need_q ? nullptr : m->q, tc ? m->qb : nullptr, 1.0f, write_kv,
                      m->stream, &sv, write_kv ? r.rows_out : nullptr);
  return launch_check(m, 1);
}

kvr_status layer_qkv(kvr_model *m, const Rows &r, int l, bool write_kv, bool keep_qkv = false,
                     bool need_q = false) {
  const Dims &dm = m->dims;
  const LayerW &w = m->layers[l];
  KVR_TRY(norm(m, w.attn_norm, r.M));
  SplitView sv;
  KVR_TRY(gemm(m, P_GEMM_QKV, m->a, w.wqkv, w.tc_qkv ? &w.tm_qkv : nullptr, w.bqkv, m->qkv, r.M,
               dm.Nqkv(), dm.d, GEMM_EPI_STORE, keep_qkv ? nullptr : &sv));
  return rope(m, r, l, write_kv, need_q, sv);
}

// Attention of layer l (after its RoPE and K/V write) into m->attn.
kvr_status attention(kvr_model *m, const Rows &r, int l) {
  const Dims &dm = m->dims;
  const LayerW &w = m->layers[l];
  {
    int64_t kv_bytes = (int64_t)(r.max_pos + 1) * dm.G * dm.dh * 2 * (int64_t)dm.es();
    Prof pr(m, P_ATTN, kv_bytes);
    if (r.tc5) {
      static const CUtensorMap unused{};  // a batch's views come from r.tmaps
      const char *e = launch_attention_tc5(
          m->qb, r.pos, r.blocks, r.n_blocks, r.n_splits, dm, l, r.single.pages, r.single.table,
          r.tm_kv ? *r.tm_kv : unused, m->attn_ws_o, m->attn_ws_ml, m->attn, m->dev_flag,
          m->stream, r.tmaps ? r.views : nullptr, r.tmaps);
      if (!e)
        e = launch_attention_combine(r.blocks, r.n_blocks, r.max_block_rows, r.n_splits, dm,
                                     m->attn_ws_o, m->attn_ws_ml, m->attn, m->stream,
                                     w.tc_o ? w.wo : nullptr,
                                     (long long)dm.d * dm.H * dm.dh * (long long)dm.es());
      if (e) return fail(KVR_E_CUDA, "attention: %s", e);
      KVR_TRY(launch_check(m, r.n_splits > 1 ? 2 : 1));
    } else if (use_tc_attention(m)) {
      const char *e = launch_attention_tc(m->qb, r.pos, r.blocks, r.n_blocks, r.max_block_rows,
                                          r.n_splits, dm, l, r.views, r.single, m->attn_ws_o,
                                          m->attn_ws_ml, m->attn, m->stream);
      if (e) return fail(KVR_E_CUDA, "attention: %s", e);
      KVR_TRY(launch_check(m, r.n_splits > 1 ? 2 : 1));
    } else {
      launch_attention_simt(m->q, r.pos, r.M, dm, l, r.views, r.rowdoc, r.single, m->attn,
                            m->stream);
      KVR_TRY(launch_check(m, 1));
    }
  }
  return KVR_OK;
}

// Attention, O projection, MLP of layer l (after layer_qkv).
kvr_status layer_rest(kvr_model *m, const Rows &r, int l) {
  const Dims &dm = m->dims;
  const LayerW &w = m->layers[l];
  KVR_TRY(attention(m, r, l));
  KVR_TRY(gemm(m, P_GEMM_O, m->attn, w.wo, w.tc_o ? &w.tm_o : nullptr, nullptr, m->h, r.M, dm.d,
               dm.H * dm.dh, GEMM_EPI_ACCUM, &m->pending));
  KVR_TRY(norm(m, w.mlp_norm, r.M));
  // gate/up reduces its own split tiles (SwiGLU needs the complete sums; a
  // separate reduction kernel measured slower than the in-GEMM fixup)
  KVR_TRY(gemm(m, P_GEMM_GU, m->a, w.wgu, w.tc_gu ? &w.tm_gu : nullptr, nullptr, nullptr, r.M,
               2 * dm.F, dm.d, GEMM_EPI_SWIGLU));
  KVR_TRY(gemm(m, P_GEMM_DOWN, m->act, w.wd, w.tc_d ? &w.tm_d : nullptr, nullptr, m->h, r.M, dm.d,
               dm.F, GEMM_EPI_ACCUM, &m->pending));
  return KVR_OK;
}

// Operator R over rows r: every layer, K/V of all rows written before any of
// them attends at that layer.  kv_only: the pass produces K/V alone (prefill,
// repair), so the last layer stops after its K/V are written -- K/V of layer l
// are projections of the layer's input, and the last layer's attention and
// MLP feed only the final hidden state, which the logits passes need.
// Whether the pass's GEMMs and norms can run as chains (launch_gemm_chain):
// every projection on the tensor cores, rows no more than the SMs, the
// residual width within the chain norm's reach.
bool chain_ok(const kvr_model *m, const Rows &r) {
  const Dims &dm = m->dims;
  if (!m->use_chain || !m->chain_bar || !m->use_tc || !m->defer_splits || r.rows_out ||
      dm.dtype != KVR_DTYPE_BF16 || r.M <= 0 || r.M > m->num_sms || dm.d > 4096 || dm.d % 4)
    return false;
  for (int l = 0; l < dm.L; ++l) {
    const LayerW &w = m->layers[l];
    if (!w.tc_qkv || !w.tc_o || !w.tc_gu || !w.tc_d) return false;
  }
  return true;
}

// The pass with the projections and norms in chains, one launch per layer
// boundary: [norm, QKV] of layer 0, then after each layer's attention
// [O, norm, gate/up, down] and the next layer's [norm, QKV].  RoPE and the
// attention stay kernels of their own.
kvr_status run_pass_chain(kvr_model *m, const Rows &r, bool kv_only) {
  const Dims &dm = m->dims;
  const size_t words = gemm_chain_bar_words();
  if (cudaMemsetAsync(m->chain_bar, 0, (size_t)(dm.L + 1) * words * sizeof(unsigned),
                      m->stream) != cudaSuccess)
    return fail(KVR_E_CUDA, "chain counters");
  KVR_TRY(embed(m, r));
  auto norm_step = [&](const float *gain) {
    ChainStep st;
    st.norm = true;
    st.h = m->h;
    st.gain = gain;
    st.eps = (float)dm.eps;
    st.d = dm.d;
    st.out = m->a;
    return st;
  };
  auto gemm_step = [&](const void *X, const void *W, const CUtensorMap *tm, const float *bias,
                       float *Y, int N, int K, int epi, bool defer) {
    ChainStep st;
    st.g = GemmArgs{X, W, bias, Y, r.M, N, K, K, N, dm.dtype, epi == GEMM_EPI_ACCUM};
    st.tmW = tm;
    st.epi = epi;
    st.out2 = epi == GEMM_EPI_SWIGLU ? m->act : nullptr;
    st.ld2 = N / 2;
    st.defer = defer;
    return st;
  };
  auto qkv_step = [&](int l) {
    const LayerW &w = m->layers[l];
    return gemm_step(m->a, w.wqkv, &w.tm_qkv, w.bqkv, m->qkv, dm.Nqkv(), dm.d, GEMM_EPI_STORE,
                     true);
  };
  int ci = 0;
  auto run = [&](const std::vector<ChainStep> &st, SplitView *last) -> kvr_status {
    int64_t bytes = 0;
    for (const ChainStep &x : st)
      if (!x.norm) bytes += (int64_t)x.g.N * x.g.K * dm.es();
    Prof pr(m, P_GEMM_CHAIN, bytes);
    const char *e = launch_gemm_chain(st.data(), (int)st.size(), m->tcw,
                                      m->chain_bar + (size_t)ci * words, m->stream, last);
    ++ci;
    if (e) return fail(KVR_E_CUDA, "GEMM chain (%d steps): %s", (int)st.size(), e);
    return launch_check(m, 1);
  };
  SplitView sv;
  KVR_TRY(run({norm_step(m->layers[0].attn_norm), qkv_step(0)}, &sv));
  for (int l = 0; l < dm.L; ++l) {
    const LayerW &w = m->layers[l];
    KVR_TRY(rope(m, r, l, true, false, sv));
    if (kv_only && l + 1 == dm.L) break;
    KVR_TRY(attention(m, r, l));
    std::vector<ChainStep> st = {
        gemm_step(m->attn, w.wo, &w.tm_o, nullptr, m->h, dm.d, dm.H * dm.dh, GEMM_EPI_ACCUM, true),
        norm_step(w.mlp_norm),
        gemm_step(m->a, w.wgu, &w.tm_gu, nullptr, nullptr, 2 * dm.F, dm.d, GEMM_EPI_SWIGLU, false),
        gemm_step(m->act, w.wd, &w.tm_d, nullptr, m->h, dm.d, dm.F, GEMM_EPI_ACCUM, true)};
    if (l + 1 < dm.L) {
      st.push_back(norm_step(m->layers[l + 1].attn_norm));
      st.push_back(qkv_step(l + 1));
      KVR_TRY(run(st, &sv));
    } else {
      KVR_TRY(run(st, &m->pending));  // the final norm adds the down projection's split tiles
    }
  }
  return KVR_OK;
}

// With rows_out: after layer l's RoPE, at the end of each group of rd_every
// layers, the event the group's host copies wait on.  Inside a capture the
// event is recorded on a side branch (rd_cap), so that the pass's kernels
// keep their programmatic edges; the branch rejoins at the end of the pass.
kvr_status rows_ready(kvr_model *m, const Rows &r, int l, bool capturing) {
  const int L = m->dims.L;
  if (!r.rows_out || ((l + 1) % r.rd_every && l + 1 < L)) return KVR_OK;
  const int g = l / r.rd_every;
  cudaError_t e;
  if (capturing) {
    e = cudaEventRecord(m->rd_fork[g], m->stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(m->rd_cap, m->rd_fork[g], 0);
    if (e == cudaSuccess)
      e = cudaEventRecordWithFlags(m->rd_ev[g], m->rd_cap, cudaEventRecordExternal);
  } else {
    e = cudaEventRecord(m->rd_ev[g], m->stream);
  }
  return e == cudaSuccess ? KVR_OK : fail(KVR_E_CUDA, "readback event: %s", cudaGetErrorString(e));
}

kvr_status run_pass(kvr_model *m, const Rows &r, bool kv_only) {
  if (r.M <= 0) return KVR_OK;
  if (chain_ok(m, r)) return run_pass_chain(m, r, kv_only);
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (r.rows_out) CUDA_TRY(cudaStreamIsCapturing(m->stream, &cs));
  const bool capturing = cs == cudaStreamCaptureStatusActive;
  KVR_TRY(embed(m, r));
  for (int l = 0; l < m->dims.L; ++l) {
    KVR_TRY(layer_qkv(m, r, l, true));
    KVR_TRY(rows_ready(m, r, l, capturing));
    if (!kv_only || l + 1 < m->dims.L) KVR_TRY(layer_rest(m, r, l));
  }
  if (capturing) {
    CUDA_TRY(cudaEventRecord(m->rd_join, m->rd_cap));
    CUDA_TRY(cudaStreamWaitEvent(m->stream, m->rd_join, 0));
  }
  return KVR_OK;
}

// The repair pass through a CUDA graph: the launch sequence of a pass
// depends only on the cache, the row count and the attention block/split
// plan (positions, tokens and block contents are read from device memory),
// so it is captured once per such key and replayed.  Only on a stream that
// can be captured (not the legacy default stream) and with profiling off.
kvr_status run_pass_graph(kvr_model *m, kvr_cache *c, const Rows &r) {
  if (!m->use_graphs || m->prof || m->stream == nullptr) return run_pass(m, r, true);
  for (auto &g : c->graphs)
    if (g.M == r.M && g.nb == r.n_blocks && g.ns == r.n_splits && g.rows_out == r.rows_out) {
      cudaError_t e = cudaGraphLaunch(g.exec, m->stream);
      if (e != cudaSuccess) return fail(KVR_E_CUDA, "graph launch: %s", cudaGetErrorString(e));
      m->launches += g.kernels;
      return KVR_OK;
    }
  int64_t l0 = m->launches;
  cudaError_t e = cudaStreamBeginCapture(m->stream, cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) return fail(KVR_E_CUDA, "begin capture: %s", cudaGetErrorString(e));
  kvr_status st = run_pass(m, r, true);
  cudaGraph_t graph = nullptr;
  e = cudaStreamEndCapture(m->stream, &graph);
  if (st || e != cudaSuccess) {
    if (graph) cudaGraphDestroy(graph);
    cudaGetLastError();
    return st ? st : fail(KVR_E_CUDA, "end capture: %s", cudaGetErrorString(e));
  }
  cudaGraphExec_t exec = nullptr;
  e = cudaGraphInstantiate(&exec, graph, 0);
  cudaGraphDestroy(graph);
  if (e != cudaSuccess) return fail(KVR_E_CUDA, "graph instantiate: %s", cudaGetErrorString(e));
  c->graphs.push_back({r.M, r.n_blocks, r.n_splits, r.rows_out, m->launches - l0, exec});
  e = cudaGraphLaunch(exec, m->stream);
  if (e != cudaSuccess) return fail(KVR_E_CUDA, "graph launch: %s", cudaGetErrorString(e));
  return KVR_OK;
}

kvr_status sync_model(kvr_model *m) {
  // the flag's copy joins the stream's work: one round trip to the host
  cudaError_t e = cudaMemcpyAsync(m->flag_h, m->dev_flag, sizeof(int), cudaMemcpyDeviceToHost,
                                  m->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(m->stream);
  if (e != cudaSuccess) return fail(KVR_E_CUDA, "device error: %s", cudaGetErrorString(e));
  const int flag = *m->flag_h;
  if (flag) {
    cudaMemset(m->dev_flag, 0, sizeof(int));
    if (m->tcw.counters)
      cudaMemset(m->tcw.counters, 0, 2 * (size_t)m->tcw.max_tiles * sizeof(int));
    return fail(KVR_E_DEVICE_TIMEOUT, "a bounded device wait ran out (code %d)", flag);
  }
  return KVR_OK;
}

// Model-owned scratch that only grows: a call that fits reuses the buffer, so
// repeated calls make no device allocation (and no cudaFree, which waits for
// the whole device).
kvr_status grow_scratch(kvr_model *m, void *&buf, size_t &have, size_t need, const char *what) {
  if (need <= have) return KVR_OK;
  CUDA_TRY(cudaStreamSynchronize(m->stream));  // the old buffer may still be in use
  dev_free(buf);
  buf = dev_alloc(need);
  have = buf ? need : 0;
  if (!buf) return fail(KVR_E_NOMEM, "%s: %zu bytes", what, need);
  return KVR_OK;
}

kvr_status use_device(const kvr_model *m) {
  CUDA_TRY(cudaSetDevice(m->device));
  return KVR_OK;
}

// ------------------------------------------------------------ weights

struct Region {
  size_t off, bytes;
};

double weight_scale() { return 0.02 / std::sqrt((65536.0 * 65536.0 - 1.0) / 3.0); }

uint64_t host_mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
uint64_t stream_out(uint64_t seed, uint64_t i) {
  return host_mix64(seed + (i + 1) * 0x9E3779B97F4A7C15ull);
}

enum Tid { T_EMBED = 0, T_LMHEAD = 1 };
int layer_tid(int l, int k) { return 8 + 16 * l + k; }
enum LayerTid { LT_WQ = 0, LT_WK, LT_WV, LT_WO, LT_WG, LT_WU, LT_WD, LT_BQ, LT_BK, LT_BV };

float bf16_bits_to_f32(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}
uint16_t f32_to_bf16_bits(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  return (uint16_t)((u + 0x7FFFu + ((u >> 16) & 1u)) >> 16);
}

// Host vector in model dtype -> fp32 device vector.
kvr_status upload_f32(kvr_model *m, float *dst, const void *src, size_t n) {
  std::vector<float> tmp(n);
  for (size_t i = 0; i < n; ++i)
    tmp[i] = m->dims.dtype == KVR_DTYPE_BF16 ? bf16_bits_to_f32(((const uint16_t *)src)[i])
                                             : ((const float *)src)[i];
  CUDA_TRY(cudaMemcpy(dst, tmp.data(), n * 4, cudaMemcpyHostToDevice));
  return KVR_OK;
}

kvr_status upload_rows(kvr_model *m, void *dst, const void *src, size_t rows, size_t cols,
                       size_t row_off) {
  size_t es = m->dims.es();
  CUDA_TRY(cudaMemcpy((char *)dst + row_off * cols * es, src, rows * cols * es,
                      cudaMemcpyHostToDevice));
  return KVR_OK;
}

// gate (inter=1) or up (inter=2) rows into the interleaved wgu.
kvr_status upload_gu(kvr_model *m, void *wgu, const void *src, int inter) {
  const Dims &dm = m->dims;
  size_t es = dm.es(), row = (size_t)dm.d * es;
  for (int b = 0; b < dm.F / GU_BLOCK; ++b) {
    size_t drow = (size_t)b * 2 * GU_BLOCK + (inter == 2 ? GU_BLOCK : 0);
    CUDA_TRY(cudaMemcpy((char *)wgu + drow * row, (const char *)src + (size_t)b * GU_BLOCK * row,
                        GU_BLOCK * row, cudaMemcpyHostToDevice));
  }
  return KVR_OK;
}

bool valid_config(const kvr_model_config *c, std::string &why) {
  if (c->vocab < 2 || c->d_model < 1 || c->n_layers < 1 || c->n_heads < 1 || c->n_kv_heads < 1 ||
      c->ffn < 1) {
    why = "non-positive dimension";
    return false;
  }
  if (c->n_heads % c->n_kv_heads) {
    why = "n_heads must be a multiple of n_kv_heads";
    return false;
  }
  if (c->dtype != KVR_DTYPE_F32 && c->dtype != KVR_DTYPE_BF16) {
    why = "dtype must be KVR_DTYPE_F32 or KVR_DTYPE_BF16";
    return false;
  }
  if (c->max_context < 1 || c->max_rows < 64) {
    why = "max_context >= 1 and max_rows >= 64 required";
    return false;
  }
  if (!(c->rope_theta > 0) || !(c->rms_eps >= 0)) {
    why = "rope_theta > 0 and rms_eps >= 0 required";
    return false;
  }
  return true;
}

// Failure-detection probe: one thread waits for *word to turn nonzero, which
// nothing makes it do.  The wait is bounded like every device wait of the
// library, by %globaltimer (limit_ns) and, should the timer stall, by an
// iteration cap; when it runs out the thread records `code` in the model's
// device flag, as a timed-out wait in a pass kernel does, and returns.
constexpr int WAIT_PROBE_CODE = 1 << 20;
__global__ void k_wait_probe(const volatile int *word, unsigned long long limit_ns,
                             unsigned int max_iters, int *dev_flag) {
  unsigned long long t0;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  for (unsigned int it = 0; *word == 0; ++it) {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    if (t - t0 >= limit_ns || it >= max_iters) {
      atomicOr(dev_flag, WAIT_PROBE_CODE);
      return;
    }
    __nanosleep(256);
  }
}

}  // namespace

// ======================================================================== ABI

namespace kvr {
bool g_pdl = true;

void set_last_error(const char *msg) { g_err = msg; }

void *dev_alloc(size_t bytes) {
  if (bytes == 0) bytes = 16;
  if (g_alloc) return g_alloc(bytes, g_alloc_ctx);
  void *p = nullptr;
  if (cudaMalloc(&p, bytes) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return p;
}
void dev_free(void *p) {
  if (!p) return;
  if (g_free)
    g_free(p, g_alloc_ctx);
  else
    cudaFree(p);
}
}  // namespace kvr

extern "C" {

const char *kvr_last_error(void) { return g_err.c_str(); }

kvr_status kvr_set_allocator(kvr_alloc_fn alloc, kvr_free_fn free_fn, void *ctx) {
  if ((alloc == nullptr) != (free_fn == nullptr))
    return fail(KVR_E_INVAL, "allocator and free function must be set together");
  g_alloc = alloc;
  g_free = free_fn;
  g_alloc_ctx = ctx;
  return KVR_OK;
}

static void trace_release(kvr_model *m);

void kvr_model_free(kvr_model *m) {
  if (!m) return;
  cudaSetDevice(m->device);
  cudaStreamSynchronize(m->stream);
  while (!m->caches.empty()) kvr_cache_free(m->caches.back());
  trace_release(m);
  prof_collect(m);
  dev_free(m->weight_block);
  dev_free(m->ws_block);
  dev_free(m->rope);
  dev_free(m->dev_flag);
  dev_free(m->chain_bar);
  dev_free(m->tcw.partials);
  dev_free(m->read_scratch);
  dev_free(m->rows_scratch);
  for (int g = 0; g < KVR_RD_GROUPS; ++g) {
    if (m->rd_ev[g]) cudaEventDestroy(m->rd_ev[g]);
    if (m->rd_fork[g]) cudaEventDestroy(m->rd_fork[g]);
  }
  if (m->rd_join) cudaEventDestroy(m->rd_join);
  if (m->rd_stream) cudaStreamDestroy(m->rd_stream);
  if (m->rd_cap) cudaStreamDestroy(m->rd_cap);
  dev_free(m->sel_scratch);
  dev_free(m->batch_scratch);
  dev_free(m->tcw.counters);
  dev_free(m->blocks_d);
  dev_free(m->attn_ws_o);
  dev_free(m->attn_ws_ml);
  if (m->stage_h) cudaFreeHost(m->stage_h);
  if (m->rb_h) cudaFreeHost(m->rb_h);
  if (m->flag_h) cudaFreeHost(m->flag_h);
  if (m->stage_ev) cudaEventDestroy(m->stage_ev);
  delete m;
}

kvr_status kvr_model_create(const kvr_model_config *cfg, const kvr_weights *wts, uint64_t seed,
                            kvr_model **out) {
  if (!cfg || !out) return fail(KVR_E_INVAL, "NULL argument");
  *out = nullptr;
  std::string why;
  if (!valid_config(cfg, why)) return fail(KVR_E_INVAL, "invalid config: %s", why.c_str());
  if (cfg->head_dim != 64 && cfg->head_dim != 128)
    return fail(KVR_E_UNSUPPORTED, "head_dim must be 64 or 128");
  if (cfg->d_model % 4 || cfg->d_model > 8192)
    return fail(KVR_E_UNSUPPORTED, "d_model must be a multiple of 4 and at most 8192");
  if (cfg->ffn % GU_BLOCK) return fail(KVR_E_UNSUPPORTED, "ffn must be a multiple of 16");
  if (cfg->max_context > 16384) return fail(KVR_E_UNSUPPORTED, "max_context above 16384");

  kvr_model *m = new kvr_model();
  Dims &dm = m->dims;
  dm = Dims{cfg->vocab, cfg->d_model, cfg->n_layers, cfg->n_heads, cfg->n_kv_heads,
            cfg->head_dim, cfg->ffn, cfg->qkv_bias ? 1 : 0, cfg->dtype, cfg->delim_id,
            cfg->rope_theta, cfg->rms_eps, cfg->max_context, cfg->max_rows};
  cudaGetDevice(&m->device);
  {
    const char *g = getenv("KVR_DISABLE_GRAPHS");
    m->use_graphs = !(g && g[0] == '1');
    const char *df = getenv("KVR_DISABLE_DEFERRED_SPLITS");
    m->defer_splits = !(df && df[0] == '1');
    const char *t5 = getenv("KVR_DISABLE_TC5_ATTENTION");
    m->use_tc5 = !(t5 && t5[0] == '1');
    const char *pd = getenv("KVR_DISABLE_PDL");
    g_pdl = !(pd && pd[0] == '1');
    // GEMM chains are opt-in: they measured slower than separate launches
    const char *ch = getenv("KVR_ENABLE_CHAIN");
    m->use_chain = ch && ch[0] == '1';
  }
  cudaDeviceGetAttribute(&m->num_sms, cudaDevAttrMultiProcessorCount, m->device);
  m->prof_classes.resize(P_NCLASS);
  for (int i = 0; i < P_NCLASS; ++i) m->prof_classes[i].name = kProfNames[i];

  auto bail = [&](kvr_status s) {
    kvr_model_free(m);
    return s;
  };

  // ---- weight block layout
  size_t es = dm.es(), d = dm.d, V = dm.V, F = dm.F, Nq = dm.Nqkv(), HD = (size_t)dm.H * dm.dh;
  auto al = [](size_t x) { return (x + 255) / 256 * 256; };
  size_t off = 0;
  size_t o_embed = off;
  off += al(V * d * es);
  size_t o_lm = off;
  off += al(V * d * es);
  size_t o_fn = off;
  off += al(d * 4);
  std::vector<size_t> lo(dm.L);
  size_t per_layer = al(Nq * d * es) + al(Nq * 4) + al(d * HD * es) + al(2 * F * d * es) +
                     al(d * F * es) + 2 * al(d * 4);
  for (int l = 0; l < dm.L; ++l) {
    lo[l] = off;
    off += per_layer;
  }
  m->weight_bytes = off;
  m->weight_block = dev_alloc(off);
  if (!m->weight_block) return bail(fail(KVR_E_NOMEM, "weights: %zu bytes", off));
  char *wb = (char *)m->weight_block;
  m->embed = wb + o_embed;
  m->lm_head = wb + o_lm;
  m->final_norm = (float *)(wb + o_fn);
  m->layers.resize(dm.L);
  for (int l = 0; l < dm.L; ++l) {
    char *p = wb + lo[l];
    LayerW &w = m->layers[l];
    w.wqkv = p;
    p += al(Nq * d * es);
    w.bqkv = (float *)p;
    p += al(Nq * 4);
    w.wo = p;
    p += al(d * HD * es);
    w.wgu = p;
    p += al(2 * F * d * es);
    w.wd = p;
    p += al(d * F * es);
    w.attn_norm = (float *)p;
    p += al(d * 4);
    w.mlp_norm = (float *)p;
    if (!dm.qkv_bias) w.bqkv = nullptr;
  }

  cudaStream_t s = 0;
  if (!wts) {
    double sc = weight_scale();
    auto init = [&](void *dst, bool f32, int tid, int64_t rows, int64_t cols, int64_t row_off,
                    int inter) {
      launch_init_tensor(dst, dm.dtype, f32, stream_out(seed, (uint64_t)tid), sc, rows, cols,
                         row_off, inter, s);
    };
    init(m->embed, false, T_EMBED, V, d, 0, 0);
    init(m->lm_head, false, T_LMHEAD, V, d, 0, 0);
    launch_fill_f32(m->final_norm, 1.f, d, s);
    for (int l = 0; l < dm.L; ++l) {
      LayerW &w = m->layers[l];
      init(w.wqkv, false, layer_tid(l, LT_WQ), HD, d, 0, 0);
      init(w.wqkv, false, layer_tid(l, LT_WK), (int64_t)dm.G * dm.dh, d, HD, 0);
      init(w.wqkv, false, layer_tid(l, LT_WV), (int64_t)dm.G * dm.dh, d,
           HD + (int64_t)dm.G * dm.dh, 0);
      if (dm.qkv_bias) {
        init(w.bqkv, true, layer_tid(l, LT_BQ), 1, HD, 0, 0);
        init((float *)w.bqkv + HD, true, layer_tid(l, LT_BK), 1, (int64_t)dm.G * dm.dh, 0, 0);
        init((float *)w.bqkv + HD + dm.G * dm.dh, true, layer_tid(l, LT_BV), 1,
             (int64_t)dm.G * dm.dh, 0, 0);
      }
      init(w.wo, false, layer_tid(l, LT_WO), d, HD, 0, 0);
      init(w.wgu, false, layer_tid(l, LT_WG), F, d, 0, 1);
      init(w.wgu, false, layer_tid(l, LT_WU), F, d, 0, 2);
      init(w.wd, false, layer_tid(l, LT_WD), d, F, 0, 0);
      launch_fill_f32(w.attn_norm, 1.f, d, s);
      launch_fill_f32(w.mlp_norm, 1.f, d, s);
    }
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess)
      return bail(fail(KVR_E_CUDA, "weight init: %s", cudaGetErrorString(e)));
  } else {
    if (!wts->embed || !wts->lm_head || !wts->final_norm || !wts->wq || !wts->wk || !wts->wv ||
        !wts->wo || !wts->wg || !wts->wu || !wts->wd || !wts->attn_norm || !wts->mlp_norm ||
        (dm.qkv_bias && (!wts->bq || !wts->bk || !wts->bv)))
      return bail(fail(KVR_E_INVAL, "missing weight pointer"));
    kvr_status st = KVR_OK;
#define UP(x)                  \
  do {                         \
    st = (x);                  \
    if (st) return bail(st);   \
  } while (0)
    UP(upload_rows(m, m->embed, wts->embed, V, d, 0));
    UP(upload_rows(m, m->lm_head, wts->lm_head, V, d, 0));
    UP(upload_f32(m, m->final_norm, wts->final_norm, d));
    size_t GD = (size_t)dm.G * dm.dh;
    for (int l = 0; l < dm.L; ++l) {
      LayerW &w = m->layers[l];
      if (!wts->wq[l] || !wts->wk[l] || !wts->wv[l] || !wts->wo[l] || !wts->wg[l] ||
          !wts->wu[l] || !wts->wd[l] || !wts->attn_norm[l] || !wts->mlp_norm[l])
        return bail(fail(KVR_E_INVAL, "missing weight pointer in layer %d", l));
      UP(upload_rows(m, w.wqkv, wts->wq[l], HD, d, 0));
      UP(upload_rows(m, w.wqkv, wts->wk[l], GD, d, HD));
      UP(upload_rows(m, w.wqkv, wts->wv[l], GD, d, HD + GD));
      if (dm.qkv_bias) {
        UP(upload_f32(m, w.bqkv, wts->bq[l], HD));
        UP(upload_f32(m, w.bqkv + HD, wts->bk[l], GD));
        UP(upload_f32(m, w.bqkv + HD + GD, wts->bv[l], GD));
      }
      UP(upload_rows(m, w.wo, wts->wo[l], d, HD, 0));
      UP(upload_gu(m, w.wgu, wts->wg[l], 1));
      UP(upload_gu(m, w.wgu, wts->wu[l], 2));
      UP(upload_rows(m, w.wd, wts->wd[l], d, F, 0));
      UP(upload_f32(m, w.attn_norm, wts->attn_norm[l], d));
      UP(upload_f32(m, w.mlp_norm, wts->mlp_norm[l], d));
    }
#undef UP
  }

  // ---- RoPE table: cos/sin of pos * theta^(-2i/dh), angles in double
  {
    int half = dm.dh / 2, P = dm.max_ctx + KVR_QUERY_RESERVE;
    std::vector<float2> t((size_t)P * half);
    for (int p = 0; p < P; ++p)
      for (int i = 0; i < half; ++i) {
        double ang = (double)p * std::pow(dm.theta, -2.0 * i / dm.dh);
        t[(size_t)p * half + i] = make_float2((float)std::cos(ang), (float)std::sin(ang));
      }
    m->rope = (float2 *)dev_alloc(t.size() * sizeof(float2));
    if (!m->rope) return bail(fail(KVR_E_NOMEM, "rope table"));
    if (cudaMemcpy(m->rope, t.data(), t.size() * sizeof(float2), cudaMemcpyHostToDevice))
      return bail(fail(KVR_E_CUDA, "rope table upload"));
  }

  // ---- workspace
  {
    size_t R = dm.max_rows, P = dm.max_ctx + KVR_QUERY_RESERVE;
    size_t sz[] = {R * 4,          R * 4,          R * d * 4,        R * d * es,  R * Nq * 4,
                   R * HD * 4,     R * HD * es,    R * 2 * F * 4,    R * F * es,
                   (size_t)KVR_QUERY_RESERVE * V * 4,
                   P * 4,          P * 8,          P * 4,            256,         R * HD * 2};
    size_t tot = 0;
    for (size_t x : sz) tot += al(x);
    m->ws_block = dev_alloc(tot);
    if (!m->ws_block) return bail(fail(KVR_E_NOMEM, "workspace: %zu bytes", tot));
    char *p = (char *)m->ws_block;
    void *ptrs[15];
    for (int i = 0; i < 15; ++i) {
      ptrs[i] = p;
      p += al(sz[i]);
    }
    m->pos_d = (int32_t *)ptrs[0];
    m->rowdoc_d = (int32_t *)ptrs[1];
    m->h = (float *)ptrs[2];
    m->a = ptrs[3];
    m->qkv = (float *)ptrs[4];
    m->q = (float *)ptrs[5];
    m->attn = ptrs[6];
    m->gu = (float *)ptrs[7];
    m->act = ptrs[8];
    m->logits = (float *)ptrs[9];
    m->scores = (float *)ptrs[10];
    m->keys = (unsigned long long *)ptrs[11];
    m->sel_out = (int32_t *)ptrs[12];
    m->sel_count = (int32_t *)ptrs[13];
    m->qb = ptrs[14];
    m->dev_flag = (int *)dev_alloc(256);
    if (!m->dev_flag) return bail(fail(KVR_E_NOMEM, "flag"));
    cudaMemset(m->dev_flag, 0, 256);
    // hand-off counters of a pass's GEMM chains (one set per chain)
    m->chain_bar =
        (unsigned *)dev_alloc((size_t)(dm.L + 1) * gemm_chain_bar_words() * sizeof(unsigned));
    if (!m->chain_bar) return bail(fail(KVR_E_NOMEM, "chain counters"));
    // positions and tokens of a pass, plus the tables of a 256-document batch
    m->stage_cap = std::max<size_t>(R * 4, P) + 4096 +
                   256 * (sizeof(CUtensorMap) + sizeof(KVView) + sizeof(void *)) / 4;
    if (cudaMallocHost(&m->stage_h, m->stage_cap * sizeof(int32_t)) != cudaSuccess)
      return bail(fail(KVR_E_NOMEM, "pinned staging"));
    cudaEventCreateWithFlags(&m->stage_ev, cudaEventDisableTiming);
    cudaEventRecord(m->stage_ev, 0);
    bool rd_ok = cudaStreamCreateWithFlags(&m->rd_stream, cudaStreamNonBlocking) == cudaSuccess &&
                 cudaStreamCreateWithFlags(&m->rd_cap, cudaStreamNonBlocking) == cudaSuccess &&
                 cudaEventCreateWithFlags(&m->rd_join, cudaEventDisableTiming) == cudaSuccess;
    for (int g = 0; g < KVR_RD_GROUPS && rd_ok; ++g)
      rd_ok = cudaEventCreateWithFlags(&m->rd_ev[g], cudaEventDisableTiming) == cudaSuccess &&
              cudaEventCreateWithFlags(&m->rd_fork[g], cudaEventDisableTiming) == cudaSuccess;
    if (!rd_ok) return bail(fail(KVR_E_CUDA, "readback streams and events"));
    if (cudaMallocHost(&m->rb_h, ((size_t)P + 8) * sizeof(int32_t)) != cudaSuccess ||
        cudaMallocHost(&m->flag_h, sizeof(int32_t)) != cudaSuccess)
      return bail(fail(KVR_E_NOMEM, "pinned readback"));
  }
  // ---- tensor-core GEMM: workspace and weight TMA descriptors
  if (dm.dtype == KVR_DTYPE_BF16) {
    const char *env = getenv("KVR_DISABLE_TC");
    m->use_tc = !(env && env[0] == '1');
    m->tcw.num_sms = m->num_sms;
    m->tcw.max_tiles = 1 << 16;
    m->tcw.dev_flag = m->dev_flag;
    m->tcw.partials = (float *)dev_alloc(gemm_tc_ws_bytes(m->num_sms));
    m->tcw.counters = (int *)dev_alloc(2 * (size_t)m->tcw.max_tiles * sizeof(int));
    if (!m->tcw.partials || !m->tcw.counters) return bail(fail(KVR_E_NOMEM, "GEMM workspace"));
    cudaMemset(m->tcw.counters, 0, 2 * (size_t)m->tcw.max_tiles * sizeof(int));
    // each tensor-core weight goes to the GEMM's blocked layout (one 16 KB
    // block per TMA box), through a scratch buffer of the largest one
    void *tmp = nullptr;
    size_t tmp_bytes = 0;
    bool nomem = false;
    auto mk = [&](CUtensorMap *tm, void *w, int N, int K) {
      if (!m->use_tc || nomem || !make_tmap_weight(tm, w, N, K)) return false;
      const size_t bytes = (size_t)N * K * 2;
      if (bytes > tmp_bytes) {
        cudaDeviceSynchronize();
        dev_free(tmp);
        tmp = dev_alloc(bytes);
        tmp_bytes = tmp ? bytes : 0;
        if (!tmp) {
          nomem = true;
          return false;
        }
      }
      if (launch_weight_tile(w, tmp, N, K, false, m->stream) ||
          cudaMemcpyAsync(w, tmp, bytes, cudaMemcpyDeviceToDevice, m->stream) != cudaSuccess) {
        nomem = true;  // reported below
        return false;
      }
      return true;
    };
    for (int l = 0; l < dm.L; ++l) {
      LayerW &w = m->layers[l];
      w.tc_qkv = mk(&w.tm_qkv, w.wqkv, dm.Nqkv(), dm.d);
      w.tc_o = mk(&w.tm_o, w.wo, dm.d, dm.H * dm.dh);
      w.tc_gu = mk(&w.tm_gu, w.wgu, 2 * dm.F, dm.d);
      w.tc_d = mk(&w.tm_d, w.wd, dm.d, dm.F);
    }
    m->tc_lm = mk(&m->tm_lm, m->lm_head, dm.V, dm.d);
    cudaDeviceSynchronize();
    dev_free(tmp);
    if (nomem) return bail(fail(KVR_E_NOMEM, "blocked weight layout: scratch or copy failed"));
  }
  if (use_tc_attention(m)) {
    m->max_blocks = dm.max_rows + 256;
    m->attn_ws_floats = (size_t)16 << 20;  // 64 MB of split-KV partials
    m->blocks_d = (int4 *)dev_alloc((size_t)m->max_blocks * sizeof(int4));
    m->attn_ws_o = (float *)dev_alloc(m->attn_ws_floats * sizeof(float));
    m->attn_ws_ml = (float2 *)dev_alloc(m->attn_ws_floats / dm.dh * sizeof(float2));
    if (!m->blocks_d || !m->attn_ws_o || !m->attn_ws_ml)
      return bail(fail(KVR_E_NOMEM, "attention workspace"));
  }
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return bail(fail(KVR_E_CUDA, "create: %s", cudaGetErrorString(e)));
  *out = m;
  return KVR_OK;
}

kvr_status kvr_model_set_stream(kvr_model *m, void *stream) {
  if (!m) return fail(KVR_E_INVAL, "NULL model");
  m->stream = (cudaStream_t)stream;
  return KVR_OK;
}

kvr_status kvr_synchronize(kvr_model *m) {
  if (!m) return fail(KVR_E_INVAL, "NULL model");
  KVR_TRY(use_device(m));
  return sync_model(m);
}

kvr_status kvr_wait_probe(kvr_model *m, int32_t limit_us) {
  if (!m) return fail(KVR_E_INVAL, "NULL model");
  if (limit_us < 1 || limit_us > 1000000) return fail(KVR_E_RANGE, "limit_us outside [1, 1e6]");
  KVR_TRY(use_device(m));
  // word 16 of the zeroed 256-byte flag block: no kernel writes it
  const unsigned long long limit_ns = (unsigned long long)limit_us * 1000ull;
  const unsigned int max_iters = (unsigned int)(limit_ns / 64 + 4096);
  k_wait_probe<<<1, 1, 0, m->stream>>>(m->dev_flag + 16, limit_ns, max_iters, m->dev_flag);
  return launch_check(m, 1);
}

int64_t kvr_launch_count(const kvr_model *m) { return m ? m->launches : 0; }

void kvr_cache_free(kvr_cache *c) {
  if (!c) return;
  cudaSetDevice(c->model->device);
  cudaStreamSynchronize(c->model->stream);
  for (auto &g : c->graphs) cudaGraphExecDestroy(g.exec);
  auto &live = c->model->caches;
  for (size_t i = 0; i < live.size(); ++i)
    if (live[i] == c) {
      live.erase(live.begin() + i);
      break;
    }
  dev_free(c->pages);
  dev_free(c->table);
  dev_free(c->tokens_d);
  delete c;
}

int32_t kvr_cache_len(const kvr_cache *c) { return c ? c->n : -1; }

// Argument checks shared by the calls that create a cache from host tokens.
static kvr_status check_context(const kvr_model *m, const int32_t *tokens, int32_t n) {
  const Dims &dm = m->dims;
  if (n < 1 || n > dm.max_ctx) return fail(KVR_E_RANGE, "n=%d outside [1, %d]", n, dm.max_ctx);
  for (int i = 0; i < n; ++i)
    if (tokens[i] < 0 || tokens[i] >= dm.V)
      return fail(KVR_E_RANGE, "token %d at position %d outside [0, %d)", tokens[i], i, dm.V);
  return KVR_OK;
}

// A new cache of n positions holding `tokens`: zeroed pages (slots never
// written hold finite values, so a masked key meets probability 0 and never
// 0 * NaN), the identity block table, the device copy of the tokens and, for
// bf16, the TMA view of the page pool.  Enqueued on the model's stream.
static kvr_status new_cache(kvr_model *m, const int32_t *tokens, int32_t n, kvr_cache **out) {
  const Dims &dm = m->dims;
  kvr_cache *c = new kvr_cache();
  c->model = m;
  m->caches.push_back(c);
  c->n = n;
  c->cap = (n + KVR_QUERY_RESERVE + KVR_PAGE - 1) / KVR_PAGE * KVR_PAGE;
  c->n_pages = c->cap / KVR_PAGE;
  size_t page_bytes = dm.page_elems() * dm.es();
  c->pages = dev_alloc((size_t)c->n_pages * page_bytes);
  c->table = (int32_t *)dev_alloc((size_t)c->n_pages * 4);
  c->tokens_d = (int32_t *)dev_alloc((size_t)c->cap * 4);
  if (!c->pages || !c->table || !c->tokens_d) {
    kvr_cache_free(c);
    return fail(KVR_E_NOMEM, "cache of %d pages", c->n_pages);
  }
  c->tokens_h.assign(tokens, tokens + n);
  if (cudaMemsetAsync(c->pages, 0, (size_t)c->n_pages * page_bytes, m->stream)) {
    kvr_cache_free(c);
    return fail(KVR_E_CUDA, "cache clear");
  }
  if (dm.dtype == KVR_DTYPE_BF16) {
    const long long rows = (long long)c->n_pages * dm.L * 2 * dm.G * KVR_PAGE;
    c->tm_kv_ok = rows < (1ll << 31) && make_tmap_bf16(&c->tm_kv, c->pages, (int)rows, dm.dh, KVR_PAGE);
  }
  std::vector<int32_t> tab(c->n_pages);
  for (int i = 0; i < c->n_pages; ++i) tab[i] = i;
  kvr_status st = stage_h2d(m, c->table, tab.data(), tab.size());
  if (!st) st = stage_h2d(m, c->tokens_d, tokens, n);
  if (st) {
    cudaStreamSynchronize(m->stream);
    kvr_cache_free(c);
    return st;
  }
  *out = c;
  return KVR_OK;
}

kvr_status kvr_cache_load(kvr_model *m, const int32_t *tokens, int32_t n, const void *k,
                          const void *v, kvr_cache **out) {
  if (!m || !tokens || !k || !v || !out) return fail(KVR_E_INVAL, "NULL argument");
  *out = nullptr;
  KVR_TRY(check_context(m, tokens, n));
  KVR_TRY(use_device(m));
  const Dims &dm = m->dims;
  kvr_cache *c = nullptr;
  KVR_TRY(new_cache(m, tokens, n, &c));
  // positions in chunks of about 32 MB of K (and as much V) through the
  // model's readback scratch; host rows [n][L][G][dh] are contiguous per chunk
  const size_t row_b = (size_t)dm.L * dm.G * dm.dh * dm.es();
  const int chunk = (int)std::max<size_t>(1, std::min<size_t>(n, ((size_t)32 << 20) / row_b));
  auto al = [](size_t x) { return (x + 255) / 256 * 256; };
  kvr_status st = grow_scratch(m, m->read_scratch, m->read_scratch_bytes,
                               2 * al((size_t)chunk * row_b), "cache load scratch");
  char *kd = (char *)m->read_scratch, *vd = kd + al((size_t)chunk * row_b);
  for (int p0 = 0; !st && p0 < n; p0 += chunk) {
    const int cnt = std::min(chunk, n - p0);
    const size_t b = (size_t)cnt * row_b, off = (size_t)p0 * row_b;
    if (cudaMemcpyAsync(kd, (const char *)k + off, b, cudaMemcpyHostToDevice, m->stream) ||
        cudaMemcpyAsync(vd, (const char *)v + off, b, cudaMemcpyHostToDevice, m->stream)) {
      st = fail(KVR_E_CUDA, "cache load upload");
      break;
    }
    launch_cache_scatter_raw(c->view(), dm.dtype, p0, cnt, kd, vd, m->stream);
    st = launch_check(m, 1);
  }
  if (!st) st = sync_model(m);
  if (st) {
    cudaStreamSynchronize(m->stream);
    kvr_cache_free(c);
    return st;
  }
  *out = c;
  return KVR_OK;
}

kvr_status kvr_prefill(kvr_model *m, const int32_t *tokens, int32_t n, kvr_cache **out) {
  if (!m || !tokens || !out) return fail(KVR_E_INVAL, "NULL argument");
  *out = nullptr;
  const Dims &dm = m->dims;
  KVR_TRY(check_context(m, tokens, n));
  KVR_TRY(use_device(m));
  kvr_cache *c = nullptr;
  KVR_TRY(new_cache(m, tokens, n, &c));
  kvr_status st = KVR_OK;
  Rows r;
  r.tokens = c->tokens_d;
  r.single = c->view();
  r.tm_kv = c->tm_kv_ok ? &c->tm_kv : nullptr;
  std::vector<int32_t> pos;
  for (int c0 = 0; c0 < n && !st; c0 += dm.max_rows) {
    int M = std::min(dm.max_rows, n - c0);
    pos.resize(M);
    for (int i = 0; i < M; ++i) pos[i] = c0 + i;
    st = stage_h2d(m, m->pos_d, pos.data(), M);
    if (st) break;
    r.M = M;
    r.pos = m->pos_d;
    r.max_pos = c0 + M - 1;
    st = plan_attention(m, r, pos.data(), nullptr);
    if (!st) st = run_pass(m, r, true);
  }
  if (st) {
    cudaStreamSynchronize(m->stream);
    kvr_cache_free(c);
    return st;
  }
  *out = c;
  return KVR_OK;
}

namespace {
// kvr_repair, and with k_out/v_out (kvr_repair_read) the copy of the rows'
// K/V to the host overlapping the pass.
kvr_status repair_impl(kvr_cache *c, const int32_t *new_tokens, int32_t edit_start,
                       int32_t edit_len, const int32_t *positions, int32_t n_positions,
                       void *k_out, void *v_out) {
  if (!c) return fail(KVR_E_INVAL, "NULL cache");
  if (c->poisoned) return fail(KVR_E_POISONED, "cache poisoned by an earlier CUDA error");
  kvr_model *m = c->model;
  const Dims &dm = m->dims;
  if (edit_len < 0 || n_positions < 0) return fail(KVR_E_RANGE, "negative length");
  if (edit_len > 0 && !new_tokens) return fail(KVR_E_INVAL, "NULL new_tokens");
  if (n_positions > 0 && !positions) return fail(KVR_E_INVAL, "NULL positions");
  int s_end = edit_start + edit_len;
  if (edit_start < 0 || s_end > c->n)
    return fail(KVR_E_RANGE, "edit span [%d, %d) outside [0, %d)", edit_start, s_end, c->n);
  for (int i = 0; i < edit_len; ++i)
    if (new_tokens[i] < 0 || new_tokens[i] >= dm.V)
      return fail(KVR_E_RANGE, "new token %d outside [0, %d)", new_tokens[i], dm.V);
  for (int i = 0; i < n_positions; ++i) {
    if (positions[i] < s_end || positions[i] >= c->n)
      return fail(KVR_E_RANGE, "position %d outside [%d, %d)", positions[i], s_end, c->n);
    if (i && positions[i] <= positions[i - 1])
      return fail(KVR_E_RANGE, "positions not strictly increasing at %d", i);
  }
  int M = edit_len + n_positions;
  if (M > dm.max_rows) return fail(KVR_E_UNSUPPORTED, "|P|=%d above max_rows", M);
  KVR_TRY(use_device(m));
  if (M == 0) return KVR_OK;
  // a1: apply the edit (the old tokens are kept to undo it should the pass
  // fail before any device work touched the cache)
  std::vector<int32_t> P(M), old(c->tokens_h.begin() + edit_start,
                                 c->tokens_h.begin() + edit_start + edit_len);
  for (int i = 0; i < edit_len; ++i) {
    c->tokens_h[edit_start + i] = new_tokens[i];
    P[i] = edit_start + i;
  }
  for (int i = 0; i < n_positions; ++i) P[edit_len + i] = positions[i];
  kvr_status st = KVR_OK;
  bool launched = false;
  if (edit_len) st = stage_h2d(m, c->tokens_d + edit_start, new_tokens, edit_len);
  if (!st) st = stage_h2d(m, m->pos_d, P.data(), M);
  if (!st) {
    Rows r;
    r.M = M;
    r.pos = m->pos_d;
    r.tokens = c->tokens_d;
    r.single = c->view();
    r.tm_kv = c->tm_kv_ok ? &c->tm_kv : nullptr;
    r.max_pos = P[M - 1];
    st = plan_attention(m, r, P.data(), nullptr);
    const size_t row_b = (size_t)dm.L * dm.G * dm.dh * dm.es();  // one row, all layers
    if (!st && k_out) {
      st = grow_scratch(m, m->rows_scratch, m->rows_scratch_bytes, 2 * M * row_b, "row buffer");
      r.rows_out = m->rows_scratch;
      r.rd_every = (dm.L + KVR_RD_GROUPS - 1) / KVR_RD_GROUPS;
    }
    if (!st) {
      launched = true;
      st = run_pass_graph(m, c, r);
    }
    if (!st && k_out) {
      // group g's rows leave as soon as the pass has written them
      const char *kd = (const char *)r.rows_out, *vd = kd + M * row_b;
      const size_t lb = row_b / dm.L;
      for (int g = 0, l0 = 0; l0 < dm.L && !st; ++g, l0 += r.rd_every) {
        const size_t w = (size_t)(std::min(dm.L, l0 + r.rd_every) - l0) * lb;
        if (cudaStreamWaitEvent(m->rd_stream, m->rd_ev[g], 0) != cudaSuccess ||
            cudaMemcpy2DAsync((char *)k_out + l0 * lb, row_b, kd + l0 * lb, row_b, w, M,
                              cudaMemcpyDeviceToHost, m->rd_stream) != cudaSuccess ||
            cudaMemcpy2DAsync((char *)v_out + l0 * lb, row_b, vd + l0 * lb, row_b, w, M,
                              cudaMemcpyDeviceToHost, m->rd_stream) != cudaSuccess)
          st = fail(KVR_E_CUDA, "row readback");
      }
      const kvr_status s2 = sync_model(m);
      if (!st) st = s2;
      if (cudaStreamSynchronize(m->rd_stream) != cudaSuccess && !st)
        st = fail(KVR_E_CUDA, "row readback");
    }
  }
  if (st && st != KVR_E_CUDA && !launched && edit_len) {
    // refused before the pass: put the old tokens back, host and device
    std::copy(old.begin(), old.end(), c->tokens_h.begin() + edit_start);
    if (stage_h2d(m, c->tokens_d + edit_start, old.data(), edit_len)) c->poisoned = true;
  }
  if (st == KVR_E_CUDA || (st && launched)) c->poisoned = true;
  return st;
}
}  // namespace

kvr_status kvr_repair(kvr_cache *c, const int32_t *new_tokens, int32_t edit_start,
                      int32_t edit_len, const int32_t *positions, int32_t n_positions) {
  return repair_impl(c, new_tokens, edit_start, edit_len, positions, n_positions, nullptr,
                     nullptr);
}

kvr_status kvr_repair_read(kvr_cache *c, const int32_t *new_tokens, int32_t edit_start,
                           int32_t edit_len, const int32_t *positions, int32_t n_positions,
                           void *k_out, void *v_out) {
  if (edit_len + n_positions > 0 && (!k_out || !v_out))
    return fail(KVR_E_INVAL, "NULL k_out or v_out");
  return repair_impl(c, new_tokens, edit_start, edit_len, positions, n_positions, k_out, v_out);
}

kvr_status kvr_repair_batch(kvr_model *m, const kvr_repair_req *reqs, int32_t n_reqs) {
  if (!m || (n_reqs > 0 && !reqs)) return fail(KVR_E_INVAL, "NULL argument");
  if (n_reqs < 0 || n_reqs > 256) return fail(KVR_E_RANGE, "n_reqs=%d outside [0, 256]", n_reqs);
  const Dims &dm = m->dims;
  std::vector<int32_t> P, rowdoc;
  int max_pos = 0;
  // validate everything before touching any cache
  for (int r = 0; r < n_reqs; ++r) {
    const kvr_repair_req &q = reqs[r];
    if (!q.cache || q.cache->model != m) return fail(KVR_E_INVAL, "request %d: bad cache", r);
    if (q.cache->poisoned) return fail(KVR_E_POISONED, "request %d: cache poisoned", r);
    for (int s = 0; s < r; ++s)
      if (reqs[s].cache == q.cache) return fail(KVR_E_INVAL, "cache repeated in a batch");
    if (q.n_edits < 0 || q.n_positions < 0) return fail(KVR_E_RANGE, "request %d: negative", r);
    std::vector<char> inP(q.cache->n, 0);
    int tk = 0;
    for (int e = 0; e < q.n_edits; ++e) {
      int s0 = q.edit_start[e], L = q.edit_len[e];
      if (L < 0 || s0 < 0 || s0 + L > q.cache->n)
        return fail(KVR_E_RANGE, "request %d edit %d outside the context", r, e);
      for (int i = 0; i < L; ++i) {
        if (inP[s0 + i]) return fail(KVR_E_RANGE, "request %d: edits overlap", r);
        inP[s0 + i] = 1;
        int t = q.new_tokens[tk + i];
        if (t < 0 || t >= dm.V) return fail(KVR_E_RANGE, "request %d: token out of range", r);
      }
      tk += L;
    }
    for (int i = 0; i < q.n_positions; ++i) {
      int p = q.positions[i];
      if (p < 0 || p >= q.cache->n || (i && p <= q.positions[i - 1]))
        return fail(KVR_E_RANGE, "request %d: positions invalid at %d", r, i);
      if (inP[p]) return fail(KVR_E_RANGE, "request %d: position %d inside an edit", r, p);
      inP[p] = 2;
    }
    for (int p = 0; p < q.cache->n; ++p)
      if (inP[p]) {
        P.push_back(p);
        rowdoc.push_back(r);
        max_pos = std::max(max_pos, p);
      }
  }
  int M = (int)P.size();
  if (M > dm.max_rows) return fail(KVR_E_UNSUPPORTED, "sum |P|=%d above max_rows", M);
  KVR_TRY(use_device(m));
  if (M == 0) return KVR_OK;
  // apply the edits
  for (int r = 0; r < n_reqs; ++r) {
    const kvr_repair_req &q = reqs[r];
    int tk = 0;
    for (int e = 0; e < q.n_edits; ++e) {
      int s0 = q.edit_start[e], L = q.edit_len[e];
      for (int i = 0; i < L; ++i) q.cache->tokens_h[s0 + i] = q.new_tokens[tk + i];
      if (L) KVR_TRY(stage_h2d(m, q.cache->tokens_d + s0, q.new_tokens + tk, L));
      tk += L;
    }
  }
  // device tables, in the model's batch scratch (grown, never shrunk; reused
  // in stream order): the documents' TMA views of their pages (when every
  // cache has one), their cache views and token pointers
  bool all_tm = true;
  for (int r = 0; r < n_reqs; ++r) all_tm = all_tm && reqs[r].cache->tm_kv_ok;
  const size_t mb = all_tm ? (size_t)n_reqs * sizeof(CUtensorMap) : 0;
  const size_t vb = n_reqs * sizeof(KVView), tb = n_reqs * sizeof(void *);
  std::vector<int32_t> host((mb + vb + tb + 3) / 4);
  char *hb = (char *)host.data();
  for (int r = 0; r < n_reqs; ++r) {
    if (all_tm) memcpy(hb + r * sizeof(CUtensorMap), &reqs[r].cache->tm_kv, sizeof(CUtensorMap));
    const KVView v = reqs[r].cache->view();
    memcpy(hb + mb + r * sizeof(KVView), &v, sizeof(KVView));
    const int32_t *t = reqs[r].cache->tokens_d;
    memcpy(hb + mb + vb + r * sizeof(void *), &t, sizeof(void *));
  }
  KVR_TRY(grow_scratch(m, m->batch_scratch, m->batch_scratch_bytes, host.size() * 4,
                       "batch tables"));
  char *tab = (char *)m->batch_scratch;
  kvr_status st = stage_h2d(m, (int32_t *)tab, host.data(), host.size());
  if (!st) st = stage_h2d(m, m->pos_d, P.data(), M);
  if (!st) {
    // rowdoc goes through a second staging round
    st = stage_h2d(m, m->rowdoc_d, rowdoc.data(), M);
  }
  if (!st) {
    Rows r;
    r.M = M;
    r.pos = m->pos_d;
    r.rowdoc = m->rowdoc_d;
    r.views = (const KVView *)(tab + mb);
    r.doc_tokens = (const int32_t *const *)(tab + mb + vb);
    r.tmaps = all_tm ? (const CUtensorMap *)tab : nullptr;
    r.max_pos = max_pos;
    st = plan_attention(m, r, P.data(), rowdoc.data());
    if (!st) st = run_pass(m, r, true);
  }
  if (st == KVR_E_CUDA)
    for (int r = 0; r < n_reqs; ++r) reqs[r].cache->poisoned = true;
  return st;
}

kvr_status kvr_logits(kvr_model *m, const kvr_cache *c, const int32_t *query, int32_t qm,
                      float *logits_out) {
  if (!m || !c || !query || !logits_out) return fail(KVR_E_INVAL, "NULL argument");
  if (c->model != m) return fail(KVR_E_INVAL, "cache of another model");
  if (c->poisoned) return fail(KVR_E_POISONED, "cache poisoned");
  const Dims &dm = m->dims;
  if (qm < 1 || qm > KVR_QUERY_RESERVE || c->n + qm > c->cap)
    return fail(KVR_E_RANGE, "query length %d outside [1, %d]", qm, KVR_QUERY_RESERVE);
  for (int i = 0; i < qm; ++i)
    if (query[i] < 0 || query[i] >= dm.V) return fail(KVR_E_RANGE, "query token out of range");
  KVR_TRY(use_device(m));
  std::vector<int32_t> P(qm);
  for (int i = 0; i < qm; ++i) P[i] = c->n + i;
  KVR_TRY(stage_h2d(m, c->tokens_d + c->n, query, qm));
  KVR_TRY(stage_h2d(m, m->pos_d, P.data(), qm));
  Rows r;
  r.M = qm;
  r.pos = m->pos_d;
  r.tokens = c->tokens_d;
  r.single = c->view();
  r.tm_kv = c->tm_kv_ok ? &c->tm_kv : nullptr;
  r.max_pos = c->n + qm - 1;
  KVR_TRY(plan_attention(m, r, P.data(), nullptr));
  KVR_TRY(run_pass(m, r, false));
  // final RMSNorm of the last row, lm_head
  {
    Prof pr(m, P_NORM, (int64_t)dm.d * 4);
    launch_rmsnorm(m->h, m->final_norm, qm - 1, 1, dm.d, dm.eps, m->a, dm.dtype, m->stream,
                   &m->pending);
    m->pending = SplitView{};
    KVR_TRY(launch_check(m, 1));
  }
  KVR_TRY(gemm(m, P_LMHEAD, m->a, m->lm_head, m->tc_lm ? &m->tm_lm : nullptr, nullptr, m->logits,
               1, dm.V, dm.d, GEMM_EPI_STORE));
  CUDA_TRY(cudaMemcpyAsync(logits_out, m->logits, (size_t)dm.V * 4, cudaMemcpyDeviceToHost,
                           m->stream));
  return sync_model(m);
}

kvr_status kvr_select(kvr_model *m, const kvr_cache *c, kvr_policy policy, int32_t K,
                      int32_t edit_start, int32_t edit_len, const int32_t *new_tokens,
                      uint64_t seed, int32_t *positions_out, int32_t *count_out) {
  if (!m || !c || !count_out || (K > 0 && !positions_out))
    return fail(KVR_E_INVAL, "NULL argument");
  if (c->model != m) return fail(KVR_E_INVAL, "cache of another model");
  if (c->poisoned) return fail(KVR_E_POISONED, "cache poisoned");
  const Dims &dm = m->dims;
  if (K < 0) return fail(KVR_E_RANGE, "K < 0");
  if (edit_len < 0 || edit_start < 0 || edit_start + edit_len > c->n)
    return fail(KVR_E_RANGE, "edit span outside the context");
  if (edit_len > 0 && !new_tokens) return fail(KVR_E_INVAL, "NULL new_tokens");
  for (int i = 0; i < edit_len; ++i)
    if (new_tokens[i] < 0 || new_tokens[i] >= dm.V)
      return fail(KVR_E_RANGE, "new token out of range");
  if (policy < KVR_POLICY_EDITLOCAL || policy > KVR_POLICY_EDITLOCAL_BOUNDARY)
    return fail(KVR_E_INVAL, "unknown policy %d", (int)policy);
  KVR_TRY(use_device(m));
  int n = c->n, s_end = edit_start + edit_len;
  *count_out = 0;
  if (n - s_end <= 0 || K == 0) return KVR_OK;
  // scratch: the edited context, then (Attention, CacheBlend) the stale rows
  // the read-only passes overwrite and the span queries' probabilities
  auto al = [](size_t x) { return (x + 255) / 256 * 256; };
  const size_t tok_b = al((size_t)c->cap * 4);
  size_t save_b = 0, prob_b = 0;
  if (policy == KVR_POLICY_ATTENTION) {
    save_b = al((size_t)edit_len * dm.L * 2 * dm.G * dm.dh * dm.es());
    prob_b = al(attn_select_ws_bytes(edit_len, dm, n - s_end));
  } else if (policy == KVR_POLICY_CACHEBLEND) {
    save_b = al((size_t)edit_len * 2 * dm.G * dm.dh * dm.es());
  }
  if (edit_len > dm.max_rows) save_b = prob_b = 0;  // refused below
  KVR_TRY(grow_scratch(m, m->sel_scratch, m->sel_scratch_bytes, tok_b + save_b + prob_b,
                       "selector scratch"));
  char *scr = (char *)m->sel_scratch;
  int32_t *toks = (int32_t *)scr;
  kvr_status st = KVR_OK;
  if (cudaMemcpyAsync(toks, c->tokens_d, (size_t)n * 4, cudaMemcpyDeviceToDevice, m->stream))
    st = fail(KVR_E_CUDA, "token copy");
  if (!st && edit_len) st = stage_h2d(m, toks + edit_start, new_tokens, edit_len);
  int topk_k = K;
  SimpleKeys gen;  // simple policies: keys made inside the top-K kernel
  void *save = nullptr;
  void *probs = nullptr;  // Attention: the selector workspace
  if (!st && (policy == KVR_POLICY_EDITLOCAL || policy == KVR_POLICY_STRUCTURAL ||
              policy == KVR_POLICY_RANDOM || policy == KVR_POLICY_EDITLOCAL_BOUNDARY)) {
    int *bound = (int *)(m->sel_count + 1);
    if (policy == KVR_POLICY_EDITLOCAL_BOUNDARY) {
      Prof pr(m, P_SELECT, 0);
      int init = n - 1;
      st = stage_h2d(m, bound, &init, 1);
      if (!st) {
        launch_first_delim(toks, n, s_end, dm.delim, bound, m->stream);
        st = launch_check(m, 1);
      }
    }
    gen.policy = (int)policy;
    gen.tokens = toks;
    gen.delim = dm.delim;
    gen.seed = seed;
    gen.bound = bound;
    if (policy == KVR_POLICY_STRUCTURAL || policy == KVR_POLICY_EDITLOCAL_BOUNDARY) topk_k = -K;
  } else if (!st && policy == KVR_POLICY_ATTENTION) {
    if (edit_len == 0) {
      st = fail(KVR_E_RANGE, "attention policy needs a non-empty span");
    } else if (edit_len > dm.max_rows) {
      st = fail(KVR_E_UNSUPPORTED, "span above max_rows");
    } else {
      // span rows through every layer, fresh K/V written in place (saved and
      // restored), probabilities of the span queries over the stale pool keys
      std::vector<int32_t> P(edit_len);
      for (int i = 0; i < edit_len; ++i) P[i] = edit_start + i;
      save = scr + tok_b;
      probs = scr + tok_b + save_b;
      st = stage_h2d(m, m->pos_d, P.data(), edit_len);
      if (!st) {
        Rows r;
        r.M = edit_len;
        r.pos = m->pos_d;
        r.tokens = toks;
        r.single = c->view();
        r.tm_kv = c->tm_kv_ok ? &c->tm_kv : nullptr;
        r.max_pos = s_end - 1;
        st = plan_attention(m, r, P.data(), nullptr);
        launch_rows_copy(r.single, dm.dtype, r.pos, edit_len, 0, dm.L, save, true, m->stream);
        launch_fill_f32(m->scores, 0.f, (size_t)n, m->stream);
        if (!st) st = launch_check(m, 2);
        if (!st) st = embed(m, r);
        for (int l = 0; l < dm.L && !st; ++l) {
          st = layer_qkv(m, r, l, true, false, true);
          if (!st) {
            Prof pr(m, P_SELECT, 0);
            launch_attn_select_scores(m->q, edit_len, dm, l, r.single, s_end, n, probs, l == 0,
                                      m->scores, m->stream);
            st = launch_check(m, 2);
          }
          // the scores need the queries of every layer; no K/V follow the last
          if (!st && l + 1 < dm.L) st = layer_rest(m, r, l);
        }
        launch_rows_copy(r.single, dm.dtype, r.pos, edit_len, 0, dm.L, save, false, m->stream);
        if (!st) st = launch_check(m, 1);
        if (!st) {
          launch_float_keys(m->scores, n, s_end, m->keys, m->stream);
          st = launch_check(m, 1);
        }
      }
    }
  } else if (!st && policy == KVR_POLICY_CACHEBLEND) {
    if (dm.L < 2) {
      st = fail(KVR_E_UNSUPPORTED, "cacheblend needs >= 2 layers");
    } else if (edit_len == 0) {
      st = fail(KVR_E_RANGE, "cacheblend policy needs a non-empty span");
    } else if (edit_len > dm.max_rows) {
      st = fail(KVR_E_UNSUPPORTED, "span above max_rows");
    } else {
      std::vector<int32_t> P(edit_len);
      for (int i = 0; i < edit_len; ++i) P[i] = edit_start + i;
      save = scr + tok_b;
      Rows r;
      r.tokens = toks;
      r.single = c->view();
      r.tm_kv = c->tm_kv_ok ? &c->tm_kv : nullptr;
      if (!st) st = stage_h2d(m, m->pos_d, P.data(), edit_len);
      if (!st) {
        // refresh the span's layer-0 K/V (saved and restored afterwards)
        r.M = edit_len;
        r.pos = m->pos_d;
        r.max_pos = s_end - 1;
        launch_rows_copy(r.single, dm.dtype, r.pos, edit_len, 0, 1, save, true, m->stream);
        launch_fill_f32(m->scores, 0.f, (size_t)n, m->stream);
        st = launch_check(m, 2);
        if (!st) st = embed(m, r);
        if (!st) st = layer_qkv(m, r, 0, true);
      }
      // layer 0 for every pool row (their layer-0 K/V depend on their token
      // alone and are left as cached), then layer-1 K/V projection
      std::vector<int32_t> D;
      for (int c0 = s_end; c0 < n && !st; c0 += dm.max_rows) {
        int M = std::min(dm.max_rows, n - c0);
        D.resize(M);
        for (int i = 0; i < M; ++i) D[i] = c0 + i;
        st = stage_h2d(m, m->pos_d, D.data(), M);
        if (st) break;
        r.M = M;
        r.pos = m->pos_d;
        r.max_pos = c0 + M - 1;
        st = plan_attention(m, r, D.data(), nullptr);
        if (!st) st = embed(m, r);
        if (!st) st = layer_qkv(m, r, 0, false);
        if (!st) st = layer_rest(m, r, 0);
        if (!st) st = layer_qkv(m, r, 1, false, true);
        if (!st) {
          Prof pr(m, P_SELECT, 0);
          launch_kv_deviation(m->qkv, m->rope, r.pos, M, dm, r.single, m->scores, m->stream);
          st = launch_check(m, 1);
        }
      }
      if (save) {
        kvr_status s2 = stage_h2d(m, m->pos_d, P.data(), edit_len);
        if (!s2) {
          launch_rows_copy(r.single, dm.dtype, m->pos_d, edit_len, 0, 1, save, false, m->stream);
          s2 = launch_check(m, 1);
        }
        if (!st) st = s2;
      }
      if (!st) {
        launch_float_keys(m->scores, n, s_end, m->keys, m->stream);
        st = launch_check(m, 1);
      }
    }
  }
  if (!st) {
    Prof pr(m, P_SELECT, 0);
    // sel_out: [count][device flag][positions ...], read back in one copy
    const char *e = launch_topk(m->keys, n, s_end, topk_k, m->sel_out + 2, m->sel_out,
                                m->stream, gen, m->dev_flag, m->sel_out + 1);
    st = e ? fail(KVR_E_CUDA, "top-K over %d candidates: %s", n - s_end, e) : launch_check(m, 1);
  }
  // one readback: the count, the device error flag and up to K positions
  int32_t cnt = 0;
  if (!st) {
    const int kmax = std::min(K, n - s_end);
    int32_t *rb = m->rb_h;
    cudaError_t e = cudaMemcpyAsync(rb, m->sel_out, (size_t)(kmax + 2) * 4,
                                    cudaMemcpyDeviceToHost, m->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(m->stream);
    if (e != cudaSuccess) {
      st = fail(KVR_E_CUDA, "select readback: %s", cudaGetErrorString(e));
    } else if (rb[1]) {
      st = sync_model(m);  // reports the bounded wait that ran out and clears the flag
    } else {
      cnt = std::min(rb[0], kmax);
      std::copy(rb + 2, rb + 2 + cnt, positions_out);
    }
  }
  cudaStreamSynchronize(m->stream);
  if (!st) *count_out = cnt;
  return st;
}

kvr_status kvr_transplant(kvr_cache *dst, const kvr_cache *src, const int32_t *positions,
                          int32_t n_positions) {
  if (!dst || !src || (n_positions > 0 && !positions)) return fail(KVR_E_INVAL, "NULL argument");
  if (dst->model != src->model) return fail(KVR_E_INVAL, "caches of different models");
  if (dst == src) return fail(KVR_E_INVAL, "transplant into the source cache");
  if (dst->poisoned || src->poisoned) return fail(KVR_E_POISONED, "cache poisoned");
  if (dst->n != src->n) return fail(KVR_E_RANGE, "caches of different lengths");
  kvr_model *m = dst->model;
  if (n_positions < 0 || n_positions > m->dims.max_rows)
    return fail(KVR_E_RANGE, "n_positions outside [0, max_rows]");
  for (int i = 0; i < n_positions; ++i)
    if (positions[i] < 0 || positions[i] >= dst->n || (i && positions[i] <= positions[i - 1]))
      return fail(KVR_E_RANGE, "positions must be strictly increasing in [0, n)");
  KVR_TRY(use_device(m));
  if (n_positions == 0) return KVR_OK;
  for (int i = 0; i < n_positions; ++i) dst->tokens_h[positions[i]] = src->tokens_h[positions[i]];
  KVR_TRY(stage_h2d(m, m->pos_d, positions, n_positions));
  launch_transplant(dst->view(), src->view(), m->dims.dtype, m->pos_d, n_positions, m->stream);
  kvr_status st = launch_check(m, 1);
  // the token copies: one device-to-device copy per position keeps the
  // device tokens identical to the host mirror
  for (int i = 0; !st && i < n_positions; ++i)
    if (cudaMemcpyAsync(dst->tokens_d + positions[i], src->tokens_d + positions[i], 4,
                        cudaMemcpyDeviceToDevice, m->stream))
      st = fail(KVR_E_CUDA, "token copy");
  if (st == KVR_E_CUDA) dst->poisoned = true;
  return st;
}

kvr_status kvr_answer_logprob(kvr_model *m, const kvr_cache *c, const int32_t *prompt,
                              int32_t mp, const int32_t *answer, int32_t ma, double *out) {
  if (!m || !c || !prompt || !answer || !out) return fail(KVR_E_INVAL, "NULL argument");
  if (c->model != m) return fail(KVR_E_INVAL, "cache of another model");
  if (c->poisoned) return fail(KVR_E_POISONED, "cache poisoned");
  const Dims &dm = m->dims;
  int rows = mp + ma - 1;
  if (mp < 1 || ma < 1 || rows > KVR_QUERY_RESERVE || c->n + rows > c->cap)
    return fail(KVR_E_RANGE, "prompt + answer - 1 must be in [1, %d]", KVR_QUERY_RESERVE);
  std::vector<int32_t> feed(prompt, prompt + mp);
  feed.insert(feed.end(), answer, answer + ma - 1);
  for (int t : feed)
    if (t < 0 || t >= dm.V) return fail(KVR_E_RANGE, "token out of range");
  for (int i = 0; i < ma; ++i)
    if (answer[i] < 0 || answer[i] >= dm.V) return fail(KVR_E_RANGE, "answer token out of range");
  KVR_TRY(use_device(m));
  std::vector<int32_t> P(rows);
  for (int i = 0; i < rows; ++i) P[i] = c->n + i;
  KVR_TRY(stage_h2d(m, c->tokens_d + c->n, feed.data(), rows));
  KVR_TRY(stage_h2d(m, m->pos_d, P.data(), rows));
  Rows r;
  r.M = rows;
  r.pos = m->pos_d;
  r.tokens = c->tokens_d;
  r.single = c->view();
  r.tm_kv = c->tm_kv_ok ? &c->tm_kv : nullptr;
  r.max_pos = c->n + rows - 1;
  KVR_TRY(plan_attention(m, r, P.data(), nullptr));
  KVR_TRY(run_pass(m, r, false));
  // rows mp-1 .. mp+ma-2 predict answer[0..ma-1]
  {
    Prof pr(m, P_NORM, (int64_t)ma * dm.d * 4);
    launch_rmsnorm(m->h, m->final_norm, mp - 1, ma, dm.d, dm.eps, m->a, dm.dtype, m->stream,
                   &m->pending);
    m->pending = SplitView{};
    KVR_TRY(launch_check(m, 1));
  }
  KVR_TRY(gemm(m, P_LMHEAD, m->a, m->lm_head, m->tc_lm ? &m->tm_lm : nullptr, nullptr, m->logits,
               ma, dm.V, dm.d, GEMM_EPI_STORE));
  // answer ids staged behind the positions in the row-document slot
  KVR_TRY(stage_h2d(m, m->rowdoc_d, answer, ma));
  float *lp = m->scores;  // [ma] scratch
  launch_row_logprob(m->logits, ma, dm.V, m->rowdoc_d, lp, m->stream);
  KVR_TRY(launch_check(m, 1));
  std::vector<float> h(ma);
  CUDA_TRY(cudaMemcpyAsync(h.data(), lp, (size_t)ma * 4, cudaMemcpyDeviceToHost, m->stream));
  KVR_TRY(sync_model(m));
  double acc = 0.0;
  for (int i = 0; i < ma; ++i) acc += h[i];
  *out = acc / ma;
  return KVR_OK;
}

kvr_status kvr_margin(kvr_model *m, const kvr_cache *c, const int32_t *prompt, int32_t mp,
                      const int32_t *a_new, int32_t m_new, const int32_t *a_old, int32_t m_old,
                      double *margin_out) {
  if (!margin_out) return fail(KVR_E_INVAL, "NULL argument");
  double lp_new = 0.0, lp_old = 0.0;
  KVR_TRY(kvr_answer_logprob(m, c, prompt, mp, a_new, m_new, &lp_new));
  KVR_TRY(kvr_answer_logprob(m, c, prompt, mp, a_old, m_old, &lp_old));
  *margin_out = lp_new - lp_old;
  return KVR_OK;
}

kvr_status kvr_cache_tokens(const kvr_cache *c, int32_t *out) {
  if (!c || !out) return fail(KVR_E_INVAL, "NULL argument");
  memcpy(out, c->tokens_h.data(), (size_t)c->n * 4);
  return KVR_OK;
}

// Rows of positions, layers [l0, l1), gathered on the device into the model's
// readback scratch (grown, never shrunk) and copied to the host: widened to
// fp32 (raw false) or as stored (raw true).
kvr_status cache_read(const kvr_cache *c, const int32_t *positions, int32_t n_pos, int32_t l0,
                      int32_t l1, void *k_out, void *v_out, bool raw) {
  if (!c || (n_pos > 0 && (!positions || !k_out || !v_out)))
    return fail(KVR_E_INVAL, "NULL argument");
  kvr_model *m = c->model;
  const Dims &dm = m->dims;
  if (l0 < 0 || l1 > dm.L || l0 > l1 || n_pos < 0) return fail(KVR_E_RANGE, "layer range");
  for (int i = 0; i < n_pos; ++i)
    if (positions[i] < 0 || positions[i] >= c->cap) return fail(KVR_E_RANGE, "position");
  if (n_pos == 0 || l0 == l1) return KVR_OK;
  KVR_TRY(use_device(m));
  const size_t elems = (size_t)n_pos * (l1 - l0) * dm.G * dm.dh;
  const size_t eb = raw ? dm.es() : 4;
  auto al = [](size_t x) { return (x + 255) / 256 * 256; };
  const size_t pos_b = al((size_t)n_pos * 4), row_b = al(elems * eb);
  const size_t need = pos_b + 2 * row_b;
  KVR_TRY(grow_scratch(m, m->read_scratch, m->read_scratch_bytes, need, "readback scratch"));
  char *base = (char *)m->read_scratch;
  int32_t *pd = (int32_t *)base;
  void *kd = base + pos_b, *vd = base + pos_b + row_b;
  kvr_status st = (size_t)n_pos <= m->stage_cap ? stage_h2d(m, pd, positions, n_pos) : KVR_OK;
  if (!st && (size_t)n_pos > m->stage_cap &&
      cudaMemcpyAsync(pd, positions, (size_t)n_pos * 4, cudaMemcpyHostToDevice, m->stream))
    st = fail(KVR_E_CUDA, "positions upload");
  if (!st) {
    if (raw)
      launch_cache_gather_raw(c->view(), dm.dtype, pd, n_pos, l0, l1, dm.G, dm.dh, kd, vd,
                              m->stream);
    else
      launch_cache_gather(c->view(), dm.dtype, pd, n_pos, l0, l1, dm.G, dm.dh, (float *)kd,
                          (float *)vd, m->stream);
    st = launch_check(m, 1);
  }
  if (!st && (cudaMemcpyAsync(k_out, kd, elems * eb, cudaMemcpyDeviceToHost, m->stream) ||
              cudaMemcpyAsync(v_out, vd, elems * eb, cudaMemcpyDeviceToHost, m->stream)))
    st = fail(KVR_E_CUDA, "readback");
  if (!st) st = sync_model(m);
  cudaStreamSynchronize(m->stream);
  return st;
}

kvr_status kvr_cache_read(const kvr_cache *c, const int32_t *positions, int32_t n_pos,
                          int32_t l0, int32_t l1, float *k_out, float *v_out) {
  return cache_read(c, positions, n_pos, l0, l1, k_out, v_out, false);
}

kvr_status kvr_cache_read_raw(const kvr_cache *c, const int32_t *positions, int32_t n_pos,
                              int32_t l0, int32_t l1, void *k_out, void *v_out) {
  return cache_read(c, positions, n_pos, l0, l1, k_out, v_out, true);
}

kvr_status kvr_model_read_tensor(const kvr_model *m, const char *name, int32_t layer, void *out,
                                 size_t bytes) {
  if (!m || !name || !out) return fail(KVR_E_INVAL, "NULL argument");
  const Dims &dm = m->dims;
  size_t es = dm.es(), d = dm.d, HD = (size_t)dm.H * dm.dh, GD = (size_t)dm.G * dm.dh;
  std::string nm(name);
  bool per_layer = !(nm == "embed" || nm == "lm_head" || nm == "final_norm");
  if (per_layer && (layer < 0 || layer >= dm.L)) return fail(KVR_E_RANGE, "layer");
  KVR_TRY(use_device(m));
  const LayerW *w = per_layer ? &m->layers[layer] : nullptr;
  auto need = [&](size_t b) { return bytes < b ? fail(KVR_E_RANGE, "need %zu bytes", b) : KVR_OK; };
  auto rows_out = [&](const void *src, size_t rows, size_t cols, size_t row_off) -> kvr_status {
    KVR_TRY(need(rows * cols * es));
    CUDA_TRY(cudaMemcpy(out, (const char *)src + row_off * cols * es, rows * cols * es,
                        cudaMemcpyDeviceToHost));
    return KVR_OK;
  };
  // a tensor-core weight [N][K] is stored blocked: back to row-major first
  void *plain = nullptr;
  auto untiled = [&](const void *src, bool tiled, int N, int K) -> const void * {
    if (!tiled) return src;
    plain = dev_alloc((size_t)N * K * es);
    if (!plain || launch_weight_tile(src, plain, N, K, true, m->stream) ||
        cudaStreamSynchronize(m->stream) != cudaSuccess)
      return nullptr;
    return plain;
  };
  struct Freer {
    void *&p;
    ~Freer() { dev_free(p); }
  } freer{plain};
  auto vec_out = [&](const float *src, size_t n) -> kvr_status {
    KVR_TRY(need(n * es));
    std::vector<float> t(n);
    CUDA_TRY(cudaMemcpy(t.data(), src, n * 4, cudaMemcpyDeviceToHost));
    for (size_t i = 0; i < n; ++i) {
      if (es == 2)
        ((uint16_t *)out)[i] = f32_to_bf16_bits(t[i]);
      else
        ((float *)out)[i] = t[i];
    }
    return KVR_OK;
  };
  if (nm == "embed") return rows_out(m->embed, dm.V, d, 0);
  const void *src = nullptr;
  auto readable = [&](const void *p) -> kvr_status {
    return p ? KVR_OK : fail(KVR_E_NOMEM, "untiling %s", name);
  };
  if (nm == "lm_head") {
    KVR_TRY(readable(src = untiled(m->lm_head, m->tc_lm, dm.V, (int)d)));
    return rows_out(src, dm.V, d, 0);
  }
  if (nm == "final_norm") return vec_out(m->final_norm, d);
  if (nm == "wq" || nm == "wk" || nm == "wv") {
    KVR_TRY(readable(src = untiled(w->wqkv, w->tc_qkv, dm.Nqkv(), (int)d)));
    if (nm == "wq") return rows_out(src, HD, d, 0);
    if (nm == "wk") return rows_out(src, GD, d, HD);
    return rows_out(src, GD, d, HD + GD);
  }
  if (nm == "wo") {
    KVR_TRY(readable(src = untiled(w->wo, w->tc_o, (int)d, (int)HD)));
    return rows_out(src, d, HD, 0);
  }
  if (nm == "wd") {
    KVR_TRY(readable(src = untiled(w->wd, w->tc_d, (int)d, dm.F)));
    return rows_out(src, d, dm.F, 0);
  }
  if (nm == "attn_norm") return vec_out(w->attn_norm, d);
  if (nm == "mlp_norm") return vec_out(w->mlp_norm, d);
  if (nm == "bq" || nm == "bk" || nm == "bv") {
    if (!dm.qkv_bias) return fail(KVR_E_INVAL, "model has no QKV bias");
    size_t o = nm == "bq" ? 0 : (nm == "bk" ? HD : HD + GD);
    return vec_out(w->bqkv + o, nm == "bq" ? HD : GD);
  }
  if (nm == "wg" || nm == "wu") {
    KVR_TRY(need((size_t)dm.F * d * es));
    KVR_TRY(readable(src = untiled(w->wgu, w->tc_gu, 2 * dm.F, (int)d)));
    size_t row = d * es;
    for (int b = 0; b < dm.F / GU_BLOCK; ++b) {
      size_t srow = (size_t)b * 2 * GU_BLOCK + (nm == "wu" ? GU_BLOCK : 0);
      CUDA_TRY(cudaMemcpy((char *)out + (size_t)b * GU_BLOCK * row,
                          (const char *)src + srow * row, GU_BLOCK * row,
                          cudaMemcpyDeviceToHost));
    }
    return KVR_OK;
  }
  return fail(KVR_E_INVAL, "unknown tensor '%s'", name);
}

kvr_status kvr_linear(kvr_model *m, const char *name, int32_t layer, const void *x, int32_t M,
                      float *y) {
  if (!m || !name || !x || !y) return fail(KVR_E_INVAL, "NULL argument");
  const Dims &dm = m->dims;
  if (M < 1 || M > dm.max_rows) return fail(KVR_E_RANGE, "M=%d outside [1, max_rows]", M);
  std::string nm(name);
  bool per_layer = nm != "lm_head";
  if (per_layer && (layer < 0 || layer >= dm.L)) return fail(KVR_E_RANGE, "layer");
  const LayerW *w = per_layer ? &m->layers[layer] : nullptr;
  const void *W = nullptr;
  const CUtensorMap *tm = nullptr;
  const float *bias = nullptr;
  int N = 0, K = 0, epi = GEMM_EPI_STORE, cls = P_GEMM_QKV;
  if (nm == "wqkv") {
    W = w->wqkv, tm = w->tc_qkv ? &w->tm_qkv : nullptr, bias = w->bqkv, N = dm.Nqkv(), K = dm.d;
  } else if (nm == "wo") {
    W = w->wo, tm = w->tc_o ? &w->tm_o : nullptr, N = dm.d, K = dm.H * dm.dh, cls = P_GEMM_O;
  } else if (nm == "wd") {
    W = w->wd, tm = w->tc_d ? &w->tm_d : nullptr, N = dm.d, K = dm.F, cls = P_GEMM_DOWN;
  } else if (nm == "wgu") {
    W = w->wgu, tm = w->tc_gu ? &w->tm_gu : nullptr, N = 2 * dm.F, K = dm.d;
    epi = GEMM_EPI_SWIGLU, cls = P_GEMM_GU;
  } else if (nm == "lm_head") {
    W = m->lm_head, tm = m->tc_lm ? &m->tm_lm : nullptr, N = dm.V, K = dm.d, cls = P_LMHEAD;
  } else {
    return fail(KVR_E_INVAL, "unknown projection '%s'", name);
  }
  KVR_TRY(use_device(m));
  size_t es = dm.es(), xb = (size_t)M * K * es;
  size_t yn = epi == GEMM_EPI_SWIGLU ? (size_t)M * dm.F : (size_t)M * N;
  void *xd = dev_alloc(xb);
  float *yd = (float *)dev_alloc(yn * 4);
  kvr_status st = KVR_OK;
  if (!xd || !yd) st = fail(KVR_E_NOMEM, "linear buffers");
  if (!st && cudaMemcpyAsync(xd, x, xb, cudaMemcpyHostToDevice, m->stream))
    st = fail(KVR_E_CUDA, "x upload");
  if (!st) st = gemm(m, cls, xd, W, tm, bias, yd, M, N, K, epi);
  if (!st && epi == GEMM_EPI_SWIGLU) {
    // act is in the model dtype: widen on the host
    std::vector<uint8_t> tmp(yn * es);
    if (cudaMemcpyAsync(tmp.data(), m->act, yn * es, cudaMemcpyDeviceToHost, m->stream) ||
        cudaStreamSynchronize(m->stream))
      st = fail(KVR_E_CUDA, "readback");
    for (size_t i = 0; !st && i < yn; ++i)
      y[i] = es == 2 ? bf16_bits_to_f32(((uint16_t *)tmp.data())[i]) : ((float *)tmp.data())[i];
  } else if (!st) {
    if (cudaMemcpyAsync(y, yd, yn * 4, cudaMemcpyDeviceToHost, m->stream))
      st = fail(KVR_E_CUDA, "readback");
  }
  if (!st) st = sync_model(m);
  cudaStreamSynchronize(m->stream);
  dev_free(xd);
  dev_free(yd);
  return st;
}

static cudaError_t trace_attach_all(const TraceBuf &b) {
  cudaError_t e = trace_attach_rows(b);
  if (e == cudaSuccess) e = trace_attach_gemm(b);
  if (e == cudaSuccess) e = trace_attach_attn(b);
  if (e == cudaSuccess) e = trace_attach_attn5(b);
  if (e == cudaSuccess) e = trace_attach_select(b);
  return e;
}

static void trace_release(kvr_model *m) {
  if (!m->trace.rec) return;
  trace_attach_all(TraceBuf{});
  dev_free(m->trace.rec);
  dev_free(m->trace.count);
  m->trace = TraceBuf{};
}

kvr_status kvr_trace_enable(kvr_model *m, int32_t capacity) {
  if (!m || capacity < 0) return fail(KVR_E_INVAL, "NULL model or negative capacity");
#ifndef KVR_TRACE
  if (capacity > 0)
    return fail(KVR_E_UNSUPPORTED, "library built without the device trace (KVR_TRACE build)");
#endif
  CUDA_TRY(cudaSetDevice(m->device));
  CUDA_TRY(cudaStreamSynchronize(m->stream));
  trace_release(m);
  if (capacity == 0) return KVR_OK;
  TraceBuf b;
  b.rec = (unsigned long long *)dev_alloc((size_t)capacity * 16 * sizeof(uint64_t));
  b.count = (unsigned int *)dev_alloc(sizeof(unsigned int));
  b.cap = (unsigned int)capacity;
  if (!b.rec || !b.count) {
    dev_free(b.rec);
    dev_free(b.count);
    return fail(KVR_E_NOMEM, "trace buffer of %d records", capacity);
  }
  CUDA_TRY(cudaMemset(b.count, 0, sizeof(unsigned int)));
  m->trace = b;
  CUDA_TRY(trace_attach_all(b));
  return KVR_OK;
}

kvr_status kvr_trace_read(kvr_model *m, uint64_t *out, int32_t cap, int32_t *n_out) {
  if (!m || !n_out || (cap > 0 && !out)) return fail(KVR_E_INVAL, "NULL argument");
  if (!m->trace.rec) return fail(KVR_E_INVAL, "no trace buffer attached");
  CUDA_TRY(cudaSetDevice(m->device));
  CUDA_TRY(cudaStreamSynchronize(m->stream));
  unsigned int n = 0;
  CUDA_TRY(cudaMemcpy(&n, m->trace.count, sizeof n, cudaMemcpyDeviceToHost));
  *n_out = (int32_t)std::min<unsigned int>(n, 0x7fffffffu);
  size_t k = std::min<size_t>({(size_t)n, (size_t)m->trace.cap, (size_t)std::max(cap, 0)});
  if (k) CUDA_TRY(cudaMemcpy(out, m->trace.rec, k * 16 * sizeof(uint64_t), cudaMemcpyDeviceToHost));
  CUDA_TRY(cudaMemset(m->trace.count, 0, sizeof(unsigned int)));
  return KVR_OK;
}

kvr_status kvr_profile_enable(kvr_model *m, int32_t enable) {
  if (!m) return fail(KVR_E_INVAL, "NULL model");
  m->prof = enable != 0;
  return KVR_OK;
}

kvr_status kvr_profile_reset(kvr_model *m) {
  if (!m) return fail(KVR_E_INVAL, "NULL model");
  prof_collect(m);
  for (auto &c : m->prof_classes) {
    c.ms = 0;
    c.launches = 0;
    c.bytes = 0;
  }
  return KVR_OK;
}

kvr_status kvr_profile_read(kvr_model *m, int32_t cap, double *ms, int64_t *launches,
                            int64_t *bytes, char *names, int32_t names_cap, int32_t *n_out) {
  if (!m || !n_out) return fail(KVR_E_INVAL, "NULL argument");
  prof_collect(m);
  int n = (int)m->prof_classes.size();
  *n_out = n;
  int w = 0;
  for (int i = 0; i < n && i < cap; ++i) {
    if (ms) ms[i] = m->prof_classes[i].ms;
    if (launches) launches[i] = m->prof_classes[i].launches;
    if (bytes) bytes[i] = m->prof_classes[i].bytes;
    if (names) {
      const std::string &s = m->prof_classes[i].name;
      if (w + (int)s.size() + 1 <= names_cap) {
        memcpy(names + w, s.c_str(), s.size() + 1);
        w += (int)s.size() + 1;
      }
    }
  }
  return KVR_OK;
}

}  // extern "C"
