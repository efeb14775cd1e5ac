"""Oracle parity at full depth and full context on the paper-shaped workloads,
in the launch configuration the benchmark times (own CUDA stream, so repair
passes run as CUDA graphs; max_context 8192, max_rows 4096).

A CPU prefill of 5000 tokens through 32 layers is out of reach, so the stale
cache both sides start from is a seeded synthetic one (``synth.kv_rows``):
the operator R of Sec. 3 (Eq. 1) is defined for any stale cache, and the
same bits reach the GPU (``kvr_cache_load``) and the oracle.  Nothing the
oracle receives comes from the CUDA path: weights and tokens are seeded,
positions are the oracle's own selections.

The oracle runs the bf16 path (every operand of a matrix product in bf16,
sums in double).  Tolerance: max|gpu - ref| / max|ref| <= 2e-2 per layer, for
K and V over the repaired rows, and for the logits -- or, where more, twice
the oracle's own null control at that depth: the same bf16 path with its
sums and residual rounded to fp32 (the arithmetic the bf16 path specifies),
compared with the double-sum run.  On these random-init models a last-bit
change of the sums grows with depth to about 2% of the largest entry by
layer 31, so at depth that measured spread, not 2e-2, is what any
implementation of the path can promise; near the input the 2e-2 bound holds.
Selections must match the oracle's top-K except where the oracle scores of
swapped positions lie within 2e-2 * max|score| of the K-th score.
"""
import os

import numpy as np
import pytest

import oracle
from paper_2609_17983_gb300 import synth

try:
    from paper_2609_17983_gb300 import kvrepair as kv
except ImportError as _e:  # pragma: no cover
    kv, _IMPORT_ERROR = None, _e

pytestmark = pytest.mark.gpu
TOL = 2e-2
STALE_SEED = 11


def rel(a, b):
    return float(np.abs(np.asarray(a, np.float64) - b).max() / max(np.abs(b).max(), 1e-30))


def check_selection(gpu_sel, ref_sel, ref_scores, band):
    gpu_sel, ref_sel = list(map(int, gpu_sel)), list(map(int, ref_sel))
    assert len(gpu_sel) == len(ref_sel)
    if gpu_sel == ref_sel:
        return
    kth = min(ref_scores[j] for j in ref_sel)
    for j in set(gpu_sel) - set(ref_sel):
        assert ref_scores[j] >= kth - band, (j, ref_scores[j], kth)
    for j in set(ref_sel) - set(gpu_sel):
        assert ref_scores[j] <= kth + band, (j, ref_scores[j], kth)


def need_host_memory(gb):
    """These checks hold a model's worth of host weights (up to ~25 GB)."""
    try:
        with open("/proc/meminfo") as f:
            avail = {ln.split(":")[0]: int(ln.split()[1]) for ln in f}["MemAvailable"] / 2**20
    except (OSError, KeyError, ValueError):
        return
    if avail < gb:
        pytest.skip(f"needs about {gb} GB of host memory, {avail:.0f} GB available")


def bench_model(cfg):
    if kv is None:
        raise _IMPORT_ERROR
    import torch
    m = kv.Model(cfg, None, seed=0, max_context=8192, max_rows=4096)
    st = torch.cuda.Stream()
    m.set_stream(st.cuda_stream)
    m._stream = st  # keep alive
    return m


def host_weights(cfg, used, n_layers=None, lm_head=False):
    """The seeded weights the device generates for model seed 0, on the host;
    the embedding table holds only the rows of the `used` tokens (the rest
    zero), which are all the oracle's passes over those tokens read."""
    oracle.set_threads(os.cpu_count() or 1)
    W = synth.weights(cfg, 0, n_layers=n_layers, embed=False, lm_head=lm_head)
    emb = np.zeros((cfg["vocab"], cfg["d_model"]), np.uint16)
    used = np.unique(np.asarray(used))
    emb[used] = synth.rows(0, synth.TID_EMBED, used, cfg["d_model"], cfg["dtype"])
    W["embed"] = emb
    return W


def oracle_cache(k, v, tokens, layers=None):
    """The oracle's cache ([L][n][G][dh] fp32 holding bf16 values) from rows
    [n][L][G][dh] of bf16 bit patterns."""
    sl = slice(None) if layers is None else slice(0, layers)
    kf = np.ascontiguousarray(synth.bf16_bits_to_f32(k[:, sl]).transpose(1, 0, 2, 3))
    vf = np.ascontiguousarray(synth.bf16_bits_to_f32(v[:, sl]).transpose(1, 0, 2, 3))
    return oracle.Cache(kf, vf, np.asarray(tokens, np.int32).copy())


def null_cfg(cfg):
    """The oracle's null control of the bf16 path: sums rounded to fp32."""
    return dict(cfg, operands="bf16_f32sums")


def compare_rows(gk, gv, ref, null, P, name):
    """GPU rows [m][L][G][dh] (fp32) against the oracle cache at positions P,
    per layer, K and V separately, each within max(TOL, 2 x the null
    control's distance from the oracle at that layer); prints the table and
    returns the worst error relative to its bound."""
    worst, lines = 0.0, []
    for l in range(gk.shape[1]):
        ek, ev = rel(gk[:, l], ref.k[l, P]), rel(gv[:, l], ref.v[l, P])
        nk, nv = rel(null.k[l, P], ref.k[l, P]), rel(null.v[l, P], ref.v[l, P])
        tk, tv = max(TOL, 2 * nk), max(TOL, 2 * nv)
        worst = max(worst, ek / tk, ev / tv)
        lines.append(f"{l}:{max(ek, ev):.4f}/{max(nk, nv):.4f}")
        assert ek <= tk and ev <= tv, (name, l, ek, ev, nk, nv)
    print(f"{name} per layer gpu/null: " + " ".join(lines))
    return worst


def test_llama8b_full_depth_repair_logits_and_margin():
    # The benchmarked workload through all 32 layers: Llama-3-8B shape,
    # n = 5000, 8-token edit at 2500, EditLocal K = 32 (40 rows).  Every
    # repaired K/V entry of every layer, the fresh-query logits over the whole
    # vocabulary, and the answer log-probabilities and margin of Eq. 2.
    need_host_memory(40)
    cfg = synth.preset("llama8b")
    w = synth.workload("llama8b")
    doc, s, new = w["doc"], w["edit_start"], w["new_tokens"]
    n, L, G, dh = len(doc), cfg["n_layers"], cfg["n_kv_heads"], cfg["head_dim"]
    k, v = synth.kv_rows(STALE_SEED, n, L, G, dh, "bf16")
    query = synth.fill_tokens(9, 8, cfg["vocab"], cfg["delim_id"])
    prompt = synth.fill_tokens(51, 4, cfg["vocab"], cfg["delim_id"])
    a_new = synth.fill_tokens(52, 2, cfg["vocab"], cfg["delim_id"])
    a_old = synth.fill_tokens(53, 2, cfg["vocab"], cfg["delim_id"])
    stale_ref = oracle.empty_cache(cfg, n)
    stale_ref.tokens[:] = doc
    A = oracle.select(cfg, None, stale_ref, "editlocal", 32, s, new)
    P = oracle.repaired_set(s, len(new), A)

    m = bench_model(cfg)
    cache = m.load_cache(doc, k, v)
    outside = np.setdiff1d(np.arange(0, n, 37), P)
    kr, vr = cache.read_raw(outside)
    assert np.array_equal(kr, k[outside]) and np.array_equal(vr, v[outside])
    assert m.select(cache, "editlocal", 32, s, new).tolist() == A.tolist()
    cache.repair(new, s, A)
    gk, gv = cache.read(P)
    kr, vr = cache.read_raw(outside)
    assert np.array_equal(kr, k[outside]) and np.array_equal(vr, v[outside])
    glog = m.logits(cache, query)
    g_new = m.answer_logprob(cache, prompt, a_new)
    g_old = m.answer_logprob(cache, prompt, a_old)
    g_margin = m.margin(cache, prompt, a_new, a_old)
    cache.close()
    m.close()

    edited = oracle.apply_edit(doc, s, new)
    W = host_weights(cfg, np.concatenate([edited[P], query, prompt, a_new, a_old]),
                     lm_head=True)
    ref = oracle.repair(cfg, W, oracle_cache(k, v, doc), new, s, A)
    null = oracle.repair(null_cfg(cfg), W, oracle_cache(k, v, doc), new, s, A)
    del k, v
    worst = compare_rows(gk, gv, ref, null, P, "llama8b")
    rlog = oracle.logits(cfg, W, ref, query)
    nlog = oracle.logits(null_cfg(cfg), W, null, query)
    tlog = max(TOL, 2 * rel(nlog, rlog))
    assert rel(glog, rlog) <= tlog, (rel(glog, rlog), rel(nlog, rlog))
    # answer log-probabilities: lp = logit(target) - logsumexp(logits), so an
    # error of at most e in every logit moves lp by at most 2e; e is the logits
    # tolerance times the largest logit of the answer rows
    bound = {}
    for name, a in (("new", a_new), ("old", a_old)):
        feed = np.concatenate([prompt, a[:-1]])
        rows = oracle.logits_all(cfg, W, ref, feed)[len(prompt) - 1:]
        bound[name] = 2 * tlog * float(np.abs(rows).max())
    r_new = oracle.answer_logprob(cfg, W, ref, prompt, a_new)
    r_old = oracle.answer_logprob(cfg, W, ref, prompt, a_old)
    assert abs(g_new - r_new) <= bound["new"], (g_new, r_new, bound)
    assert abs(g_old - r_old) <= bound["old"], (g_old, r_old, bound)
    assert abs(g_margin - (g_new - g_old)) <= 1e-12 * max(1.0, abs(g_margin))
    assert abs(g_margin - (r_new - r_old)) <= bound["new"] + bound["old"]
    print(f"llama8b full depth: worst K/V error {worst:.2f} of its bound, logits "
          f"{rel(glog, rlog):.2e} (null control {rel(nlog, rlog):.2e}), margin gpu "
          f"{g_margin:.4f} oracle {r_new - r_old:.4f} bound {bound['new'] + bound['old']:.3f}")


def test_qwen7b_full_depth_attention_selector_and_repair():
    # Qwen2.5-7B shape (QKV bias, 28/4 heads), n = 5000, 6-token edit: the
    # stale-query Attention selector (Table 1) for every K of the sweep against
    # the oracle's scores over all 28 layers, then the repair of the span plus
    # the oracle's K = 32 selection through every layer.
    need_host_memory(40)
    cfg = synth.preset("qwen7b")
    w = synth.workload("qwen7b")
    doc, s, new = w["doc"], w["edit_start"], w["new_tokens"]
    n, L, G, dh = len(doc), cfg["n_layers"], cfg["n_kv_heads"], cfg["head_dim"]
    k, v = synth.kv_rows(STALE_SEED + 1, n, L, G, dh, "bf16")
    edited = oracle.apply_edit(doc, s, new)
    D = oracle.pool(n, s, len(new))
    W = host_weights(cfg, np.concatenate([edited[s:s + len(new)], edited[D]]))
    sc, elig = oracle.scores(cfg, W, oracle_cache(k, v, doc), "attention", s, new)
    band = TOL * float(np.abs(sc[elig]).max())
    refs = {K: oracle.topk(sc, elig, K) for K in w["Ks"]}

    m = bench_model(cfg)
    cache = m.load_cache(doc, k, v)
    for K in w["Ks"]:
        check_selection(m.select(cache, "attention", K, s, new), refs[K], sc, band)
    kr, vr = cache.read_raw(np.arange(n))  # the selector leaves the cache as it was
    assert np.array_equal(kr, k) and np.array_equal(vr, v)
    del kr, vr
    A = refs[32]
    P = oracle.repaired_set(s, len(new), A)
    cache.repair(new, s, A)
    gk, gv = cache.read(P)
    cache.close()
    m.close()
    ref = oracle.repair(cfg, W, oracle_cache(k, v, doc), new, s, A)
    null = oracle.repair(null_cfg(cfg), W, oracle_cache(k, v, doc), new, s, A)
    worst = compare_rows(gk, gv, ref, null, P, "qwen7b")
    print(f"qwen7b full depth: attention selections within the tie band for K in {w['Ks']}, "
          f"worst K/V error {worst:.2f} of its bound")


def test_mistral7b_full_size_cacheblend_selector():
    # Mistral-7B shape, n = 5000 with delimiters, 10-token edit: the
    # CacheBlend-style layer-1 K/V deviation selector (Table 1) against the
    # oracle's scores over the whole pool.  The selector reads layer 0 at every
    # position up to the pool's end and layer 1 at the pool, so there the stale
    # cache holds what a prefill of C leaves (layer 0: a function of token and
    # position alone; layer 1 at the pool: the projection of the layer-0
    # output); every other entry is synthetic.
    need_host_memory(24)
    cfg = synth.preset("mistral7b")
    w = synth.workload("mistral7b")
    doc, s, new = w["doc"], w["edit_start"], w["new_tokens"]
    n, L, G, dh, d = (len(doc), cfg["n_layers"], cfg["n_kv_heads"], cfg["head_dim"],
                      cfg["d_model"])
    D = oracle.pool(n, s, len(new))
    oracle.set_threads(os.cpu_count() or 1)
    cfg2 = dict(cfg, n_layers=2)
    W2 = synth.weights(cfg2, 0, lm_head=False)
    # layer 0 of every position, as a prefill of a one-layer model that shares
    # layer 0's embedding, attention norm, W_k, W_v and RoPE (query heads and
    # MLP reduced: they do not enter layer-0 K/V)
    ly = W2["layers"][0]
    z = np.zeros
    red = dict(attn_norm=ly["attn_norm"], mlp_norm=ly["mlp_norm"], wq=ly["wq"][:G * dh],
               wk=ly["wk"], wv=ly["wv"], wo=z((d, G * dh), np.uint16),
               wg=z((16, d), np.uint16), wu=z((16, d), np.uint16), wd=z((d, 16), np.uint16))
    cfg_red = dict(cfg, n_layers=1, n_heads=G, ffn=16)
    l0 = oracle.prefill(cfg_red, dict(embed=W2["embed"], final_norm=W2["final_norm"],
                                      lm_head=None, layers=[red]), doc)
    k, v = synth.kv_rows(STALE_SEED + 2, n, L, G, dh, "bf16")
    stale = oracle_cache(k, v, doc, layers=2)
    stale.k[0], stale.v[0] = l0.k[0], l0.v[0]
    # layer 1 at the pool: the pool rows of the stale context through layer 0
    oracle.recompute(cfg2, W2, stale, doc, D)
    assert np.array_equal(stale.k[0], l0.k[0]) and np.array_equal(stale.v[0], l0.v[0])
    for l in (0, 1):
        rows = slice(None) if l == 0 else D
        k[rows, l] = synth.f32_to_bf16_bits(stale.k[l, rows])
        v[rows, l] = synth.f32_to_bf16_bits(stale.v[l, rows])
    sc, elig = oracle.scores(cfg2, W2, stale, "cacheblend", s, new)
    ref = oracle.topk(sc, elig, 32)
    band = TOL * float(np.abs(sc[elig]).max())

    m = bench_model(cfg)
    cache = m.load_cache(doc, k, v)
    got = m.select(cache, "cacheblend", 32, s, new)
    check_selection(got, ref, sc, band)
    kr, vr = cache.read_raw(np.arange(n))
    assert np.array_equal(kr, k) and np.array_equal(vr, v)  # read-only
    cache.close()
    m.close()
    print(f"mistral7b cacheblend: {len(set(got.tolist()) & set(ref.tolist()))}/32 shared with "
          f"the oracle's top-K; band {band:.3g} of scores up to {np.abs(sc[elig]).max():.3g}")
