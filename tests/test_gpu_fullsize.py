"""Full-size checks on the paper-shaped workloads, in the launch configuration
the benchmark times (own CUDA stream, so repair passes run as CUDA graphs;
max_context 8192, max_rows 4096).

The oracle cannot prefill 5000 tokens through 32 layers, so the checks are
(i) outputs the oracle computes exactly at full size -- closed-form
selections, and the layer-0 K/V of repaired rows, which depend only on each
row's token and position -- and (ii) properties that hold at any size: the
Eq. 1 endpoint identity, untouched rows outside P, idempotence, read-only
selectors, and batch == per-document repair.
"""
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


def rel(a, b):
    return float(np.abs(np.asarray(a, np.float64) - b).max() / max(np.abs(b).max(), 1e-30))


def bench_model(cfg):
    if kv is None:
        raise _IMPORT_ERROR
    import torch
    m = kv.Model(cfg, None, seed=0, max_context=8192, max_rows=4096)
    st = torch.cuda.Stream()
    m.set_stream(st.cuda_stream)
    m._stream = st  # keep alive
    return m


def layer0_reference(cfg, tokens, rows):
    """Layer-0 K/V of the given rows, exact from token and position: the
    oracle's operator R on a one-layer model writes them before attending."""
    rows = np.asarray(rows)
    used = np.unique(tokens[rows])
    remap = {int(t): i for i, t in enumerate(used)}
    W = synth.weights(cfg, 0, n_layers=1, embed=False, lm_head=False)
    W["embed"] = synth.rows(0, synth.TID_EMBED, used, cfg["d_model"], cfg["dtype"])
    ocfg = dict(cfg, n_layers=1, vocab=len(used))
    toks = np.zeros(len(tokens), np.int32)
    toks[rows] = [remap[int(t)] for t in tokens[rows]]
    c = oracle.empty_cache(ocfg, len(tokens))
    oracle.recompute(ocfg, W, c, toks, rows)
    return c.k[0, rows], c.v[0, rows]


def sample_rows(n, P, stride=11):
    s = set(range(0, n, stride)) | set(int(p) for p in P)
    for p in P:
        s |= {max(0, int(p) - 1), min(n - 1, int(p) + 1)}
    return np.array(sorted(s))


@pytest.fixture(scope="module")
def llama():
    cfg = synth.preset("llama8b")
    m = bench_model(cfg)
    yield cfg, m
    m.close()


def test_llama8b_bench_workload(llama):
    cfg, m = llama
    w = synth.workload("llama8b")
    doc, s, new = w["doc"], w["edit_start"], w["new_tokens"]
    n = len(doc)
    cache = m.prefill(doc)
    A = m.select(cache, "editlocal", 32, s, new)
    ref_cache = oracle.empty_cache(cfg, n)
    ref_cache.tokens[:] = doc
    assert A.tolist() == oracle.select(cfg, None, ref_cache, "editlocal", 32, s, new).tolist()
    P = np.concatenate([np.arange(s, s + len(new)), A])
    rows = sample_rows(n, P)
    k0, v0 = cache.read(rows)
    cache.repair(new, s, A)
    k1, v1 = cache.read(rows)
    outside = ~np.isin(rows, P)
    assert np.array_equal(k1[outside], k0[outside]) and np.array_equal(v1[outside], v0[outside])
    # layer-0 K/V of the repaired rows against the oracle
    edited = oracle.apply_edit(doc, s, new)
    rk, rv = layer0_reference(cfg, edited, P)
    gk, gv = cache.read(P, 0, 1)
    assert rel(gk[:, 0], rk) <= TOL and rel(gv[:, 0], rv) <= TOL
    # idempotence (graph replay of the same pass)
    cache.repair(new, s, A)
    k2, v2 = cache.read(rows)
    assert np.array_equal(k1, k2) and np.array_equal(v1, v2)
    cache.close()


def test_llama8b_endpoint_identity_full_size(llama):
    # Eq. 1 at the bench size: the full suffix repaired equals a prefill of
    # C' -- in bf16 up to rounding noise, which compounds with depth.  As in
    # the paper's sanity check, the noise level comes from a null control:
    # the same prefill of C' computed with a different row chunking (so only
    # the rounding order differs).  The endpoint gap must not exceed it.
    cfg, m = llama
    w = synth.workload("llama8b")
    doc, s, new = w["doc"], w["edit_start"], w["new_tokens"]
    n = len(doc)
    edited = oracle.apply_edit(doc, s, new)
    cache = m.prefill(doc)
    cache.repair(new, s, np.arange(s + len(new), n))
    fresh = m.prefill(edited)
    other = kv.Model(cfg, None, seed=0, max_context=8192, max_rows=2048)
    control = other.prefill(edited)
    rows = sample_rows(n, [], stride=7)
    k1, v1 = cache.read(rows)
    k2, v2 = fresh.read(rows)
    k3, v3 = control.read(rows)

    def l2(a, b):
        d = np.asarray(a, np.float64) - b
        return float(np.linalg.norm(d) / np.linalg.norm(b))

    for l in range(cfg["n_layers"]):
        for x, y, z in ((k1, k2, k3), (v1, v2, v3)):
            gap, noise = l2(x[:, l], y[:, l]), l2(z[:, l], y[:, l])
            assert gap <= 1.25 * noise + 1e-4, (l, gap, noise)
    assert l2(k1[:, 0], k2[:, 0]) <= 1e-3  # layer 0 is token-only: near exact
    control.close()
    other.close()
    cache.close()
    fresh.close()


def test_qwen7b_selectors_and_repair():
    cfg = synth.preset("qwen7b")
    m = bench_model(cfg)
    w = synth.workload("qwen7b")
    doc, s, new = w["doc"], w["edit_start"], w["new_tokens"]
    n = len(doc)
    cache = m.prefill(doc)
    ref_cache = oracle.empty_cache(cfg, n)
    ref_cache.tokens[:] = doc
    rows = sample_rows(n, np.arange(s, s + 200), stride=17)
    k0, v0 = cache.read(rows)
    for K in w["Ks"]:
        for pol, seeds in (("editlocal", [0]), ("random", range(5))):
            for seed in seeds:
                got = m.select(cache, pol, K, s, new, seed)
                assert got.tolist() == oracle.select(cfg, None, ref_cache, pol, K, s, new,
                                                     seed).tolist()
        att = m.select(cache, "attention", K, s, new)
        assert len(att) == K and len(set(att.tolist())) == K
        assert att.min() >= s + len(new) and att.max() < n and np.all(np.diff(att) > 0)
    k1, v1 = cache.read(rows)
    assert np.array_equal(k0, k1) and np.array_equal(v0, v1)  # selectors are read-only
    A = m.select(cache, "editlocal", 32, s, new)
    cache.repair(new, s, A)
    P = np.concatenate([np.arange(s, s + len(new)), A])
    rk, rv = layer0_reference(cfg, oracle.apply_edit(doc, s, new), P)
    gk, gv = cache.read(P, 0, 1)
    assert rel(gk[:, 0], rk) <= TOL and rel(gv[:, 0], rv) <= TOL
    cache.close()
    m.close()


def test_mistral7b_structural_and_cacheblend():
    cfg = synth.preset("mistral7b")
    m = bench_model(cfg)
    w = synth.workload("mistral7b")
    doc, s, new = w["doc"], w["edit_start"], w["new_tokens"]
    n = len(doc)
    cache = m.prefill(doc)
    ref_cache = oracle.empty_cache(cfg, n)
    ref_cache.tokens[:] = doc
    got = m.select(cache, "structural", 32, s, new)
    assert got.tolist() == oracle.select(cfg, None, ref_cache, "structural", 32, s, new).tolist()
    n_delims = int(np.sum(doc[s + len(new):] == cfg["delim_id"]))
    assert len(got) == min(32, n_delims)  # fewer when the pool holds fewer delimiters
    for K in (32, 4096):  # EditLocal@boundary: window to the next delimiter, K caps it
        got = m.select(cache, "editlocal_boundary", K, s, new)
        ref = oracle.select(cfg, None, ref_cache, "editlocal_boundary", K, s, new)
        assert got.tolist() == ref.tolist(), K
    rows = sample_rows(n, np.arange(s, s + 100), stride=19)
    k0, v0 = cache.read(rows)
    cb = m.select(cache, "cacheblend", 32, s, new)
    assert len(cb) == 32 and cb.min() >= s + len(new) and np.all(np.diff(cb) > 0)
    k1, v1 = cache.read(rows)
    assert np.array_equal(k0, k1) and np.array_equal(v0, v1)
    cache.repair(new, s, cb)
    P = np.concatenate([np.arange(s, s + len(new)), cb])
    rk, rv = layer0_reference(cfg, oracle.apply_edit(doc, s, new), P)
    gk, gv = cache.read(P, 0, 1)
    assert rel(gk[:, 0], rk) <= TOL and rel(gv[:, 0], rv) <= TOL
    cache.close()
    m.close()


def test_llama8b_margin_harness_endpoints(llama):
    # The margin harness (Eq. 2) at the bench size, through both operators
    # at the full-suffix endpoint.  Transplanting every row from s on gives
    # the fresh prefill's margins exactly.  Repairing the full suffix matches
    # them up to bf16 rounding noise, whose level comes from null controls:
    # the same prefill of C' tiled with other row chunkings (the margins of
    # equivalent caches spread by a few 1e-2 nats).  Over 8 answer pairs and 3
    # controls the repaired gap stays within twice the controls' RMS spread.
    cfg, m = llama
    w = synth.workload("llama8b")
    doc, s, new = w["doc"], w["edit_start"], w["new_tokens"]
    n = len(doc)
    edited = oracle.apply_edit(doc, s, new)
    prompt = synth.fill_tokens(51, 12, cfg["vocab"], cfg["delim_id"])
    pairs = [(synth.fill_tokens(52 + 2 * i, 4, cfg["vocab"], cfg["delim_id"]),
              synth.fill_tokens(53 + 2 * i, 4, cfg["vocab"], cfg["delim_id"])) for i in range(8)]
    stale, fresh = m.prefill(doc), m.prefill(edited)
    rep, trans = m.prefill(doc), m.prefill(doc)
    rep.repair(new, s, np.arange(s + len(new), n))
    trans.transplant_from(fresh, np.arange(s, n))
    rows = sample_rows(n, [], stride=13)
    kt, vt = trans.read(rows)
    kf, vf = fresh.read(rows)
    after = rows >= s
    assert np.array_equal(kt[after], kf[after]) and np.array_equal(vt[after], vf[after])
    assert np.array_equal(trans.tokens(), edited)

    def margins(model, cache):
        return np.array([model.margin(cache, prompt, a, b) for a, b in pairs])

    mg = {k: margins(m, c) for k, c in dict(stale=stale, fresh=fresh, rep=rep,
                                           trans=trans).items()}
    for c in (stale, fresh, rep, trans):
        c.close()
    ctrl = []
    for max_rows in (2048, 1024, 512):
        other = kv.Model(cfg, None, seed=0, max_context=8192, max_rows=max_rows)
        control = other.prefill(edited)
        ctrl.append(margins(other, control) - mg["fresh"])
        control.close()
        other.close()
    noise = float(np.sqrt(np.mean(np.square(ctrl))))
    assert all(np.all(np.isfinite(v)) for v in mg.values())
    assert np.array_equal(mg["trans"], mg["fresh"]), mg
    gap = float(np.sqrt(np.mean(np.square(mg["rep"] - mg["fresh"]))))
    assert gap <= 2 * noise + 1e-3, (mg, noise)
    # the edit moves the margins far beyond the noise, so MR is meaningful
    shift = float(np.sqrt(np.mean(np.square(mg["fresh"] - mg["stale"]))))
    assert shift >= 5 * noise, (mg, noise)


def test_batched_repair_16x8192_matches_per_document(llama):
    # 16 documents of 8192 tokens, 4 non-overlapping edits each with an
    # edit-local window of 32 after every span, all in one batched call
    cfg, m = llama
    docs, reqs, singles = [], [], []
    for d in range(16):
        doc = synth.document(100 + d, 8192, cfg["vocab"], cfg["delim_id"])
        edits = []
        A = []
        for (st, ln) in synth.batch_edits(200 + d, 8192, 4, (2, 16), 32):
            new = synth.edit_tokens(300 + d * 7 + st, doc[st:st + ln], cfg["vocab"])
            edits.append((st, new))
            A += list(range(st + ln, st + ln + 32))
        docs.append(doc)
        reqs.append((edits, np.array(sorted(set(A)))))
    batch_caches = [m.prefill(doc) for doc in docs]
    m.repair_batch([(c, e, A) for c, (e, A) in zip(batch_caches, reqs)])
    for d in (0, 7, 15):
        single = m.prefill(docs[d])
        edits, A = reqs[d]
        # same rows through the single-document path: all edits, one pass
        toks = docs[d].copy()
        P = set(A.tolist())
        for st, new in edits:
            toks[st:st + len(new)] = new
            P |= set(range(st, st + len(new)))
        m.repair_batch([(single, edits, A)])
        rows = sample_rows(8192, sorted(P), stride=29)
        k1, v1 = batch_caches[d].read(rows)
        k2, v2 = single.read(rows)
        # the two passes tile different row counts, so they differ by bf16
        # rounding noise that compounds with depth: bounded per layer by the
        # level two equivalent prefills differ by (relative L2 <= 0.022 at
        # layer 31 in the endpoint test's null control), layer 0 near exact
        for l in range(cfg["n_layers"]):
            for x, y in ((k1[:, l], k2[:, l]), (v1[:, l], v2[:, l])):
                e = float(np.linalg.norm(x.astype(np.float64) - y) / np.linalg.norm(y))
                assert e <= (1e-3 if l == 0 else 3e-2), (d, l, e)
        assert np.array_equal(batch_caches[d].tokens(), toks)
        single.close()
    for c in batch_caches:
        c.close()
