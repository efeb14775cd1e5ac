"""Pins of the CPU oracle against facts that the paper and the mathematics fix.

Each test names what pins it: a library routine (the textbook decoder in
tests/textbook.py), an identity of Sec. 3 (Eq. 1 endpoint, upstream
invariance), a closed form of Table 1, a published test vector, or a
hand-worked golden case under tests/golden/.  None of them re-types the
oracle's own formulas.
"""
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2609_17983_gb300 import synth
from tests import textbook

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def read_golden(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            k, v = line.split(":", 1)
            out[k.strip()] = v.split()
    return out


def small_workload(dtype="fp32", n=160, s=60, L=4, seed=0, **over):
    cfg = synth.preset("tiny", dtype=dtype, **over)
    W = synth.weights(cfg, seed)
    doc = synth.document(11, n, cfg["vocab"], cfg["delim_id"])
    new = synth.edit_tokens(12, doc[s:s + L], cfg["vocab"], cfg["delim_id"])
    return cfg, W, doc, s, new


@pytest.fixture(scope="module")
def tiny():
    w = synth.workload("tiny")
    cfg = w["cfg"]
    W = synth.weights(cfg, 0)
    stale = oracle.prefill(cfg, W, w["doc"])
    return dict(w, W=W, stale=stale)


# --------------------------------------------------------------- generators

def test_splitmix64_published_vectors():
    g = read_golden("splitmix64_seed1234567.txt")
    seed = int(g["seed"][0])
    want = [int(x) for x in g["outputs"]]
    got_oracle = [oracle.splitmix64((seed + i * oracle.GOLDEN) & oracle.MASK64) for i in range(5)]
    got_synth = [int(x) for x in synth.stream_out(seed, np.arange(5))]
    assert got_oracle == want
    assert got_synth == want


def test_weight_generator_moments():
    # Irwin-Hall(4) construction: mean 0, std 0.02, bounded by 2*sqrt(3) sigma.
    x = synth.tensor(7, 3, (1 << 20,), "fp32").astype(np.float64)
    assert abs(x.mean()) < 1e-4
    assert abs(x.std() - 0.02) < 2e-4
    assert np.abs(x).max() <= 0.02 * 2 * np.sqrt(3) * (1 + 1e-6)
    # bf16 bits are the fp32 values rounded to nearest even
    b = synth.tensor(7, 3, (1 << 12,), "bf16")
    f = synth.tensor(7, 3, (1 << 12,), "fp32")
    back = synth.bf16_bits_to_f32(b)
    assert np.all(np.abs(back - f) <= np.abs(f) * 2.0 ** -8 + 1e-30)


# ------------------------------------------------- forward vs the textbook

@pytest.mark.parametrize("bias", [False, True])
def test_prefill_matches_textbook_decoder(bias):
    cfg, W, doc, s, new = small_workload(qkv_bias=bias)
    ref = textbook.forward(cfg, W, doc)
    got = oracle.prefill(cfg, W, doc)
    h = oracle.recompute(cfg, W, oracle.prefill(cfg, W, doc), doc, np.arange(len(doc)),
                         want_h=True)
    for l in range(cfg["n_layers"]):
        k = ref["layers"][l]["k"].numpy()
        v = ref["layers"][l]["v"].numpy()
        # cache entries are fp32-rounded; the textbook stays in float64
        np.testing.assert_allclose(got.k[l], k, rtol=0, atol=1e-6 * np.abs(k).max())
        np.testing.assert_allclose(got.v[l], v, rtol=0, atol=1e-6 * np.abs(v).max())
    hr = ref["h"].numpy()
    np.testing.assert_allclose(h, hr, rtol=0, atol=1e-6 * np.abs(hr).max())


@pytest.mark.parametrize("bias", [False, True])
def test_bf16_path_matches_textbook_decoder(bias):
    # The oracle's bf16 path (a bf16 model's default: every operand of a matrix
    # product rounded to bf16, the cache in bf16, sums in double) against the
    # textbook decoder with the same rounding points, made by torch's own
    # conversions, its library products and an attention written out over all
    # heads at once.  The values before each rounding agree to double
    # precision, so every rounding lands the same way: agreement to 1e-9.
    cfg, W, doc, s, new = small_workload(dtype="bf16", qkv_bias=bias)
    query = synth.fill_tokens(98, 5, cfg["vocab"], cfg["delim_id"])
    ref = textbook.forward(cfg, W, np.concatenate([doc, query]), operands="bf16")
    got = oracle.prefill(cfg, W, doc)
    n = len(doc)
    for l in range(cfg["n_layers"]):
        k = textbook.bf16(ref["layers"][l]["k"][:n]).numpy()
        v = textbook.bf16(ref["layers"][l]["v"][:n]).numpy()
        np.testing.assert_allclose(got.k[l], k, rtol=0, atol=1e-9 * np.abs(k).max())
        np.testing.assert_allclose(got.v[l], v, rtol=0, atol=1e-9 * np.abs(v).max())
    lg = oracle.logits(cfg, W, got, query)
    rl = ref["logits"][-1].numpy()
    np.testing.assert_allclose(lg, rl, rtol=0, atol=1e-9 * np.abs(rl).max())
    # and it is a different computation from the double one: at layer 0 the
    # rounded operands move K by at most a few bf16 steps
    exact = oracle.prefill(dict(cfg, operands="fp64"), W, doc)
    d0 = np.abs(exact.k[0].astype(np.float64) - got.k[0]).max()
    assert 0 < d0 <= 2.0 ** -6 * np.abs(exact.k[0]).max()
    assert not np.array_equal(exact.k[-1], got.k[-1])


def test_logits_match_textbook_decoder():
    cfg, W, doc, s, new = small_workload()
    query = synth.fill_tokens(99, 5, cfg["vocab"], cfg["delim_id"])
    stale = oracle.prefill(cfg, W, doc)
    got = oracle.logits(cfg, W, stale, query)
    ref = textbook.forward(cfg, W, np.concatenate([doc, query]))["logits"][-1].numpy()
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-6 * np.abs(ref).max())
    # the document's cache is not modified by the fresh query
    again = oracle.prefill(cfg, W, doc)
    assert np.array_equal(stale.k, again.k) and np.array_equal(stale.v, again.v)


def test_rope_relative_position_property():
    # <R_p q, R_r k> depends only on p - r, and R_0 is the identity.
    cfg, W, doc, s, new = small_workload(n=64)
    ref = textbook.forward(cfg, W, doc, want_logits=False)
    base = oracle.prefill(cfg, W, doc)
    # position 0's k equals the unrotated projection; compare with the textbook
    k0 = ref["layers"][0]["k"][0].numpy()
    np.testing.assert_allclose(base.k[0, 0], k0, rtol=0, atol=1e-6 * np.abs(k0).max())
    # shift invariance of dot products on a constant token sequence
    same = np.full(64, 77, np.int32)
    c = oracle.prefill(cfg, W, same)
    k = c.k[0].astype(np.float64)  # [n, G, dh] layer 0, all the same token
    d1 = np.einsum("gd,gd->g", k[10], k[3])
    d2 = np.einsum("gd,gd->g", k[40], k[33])
    np.testing.assert_allclose(d1, d2, rtol=1e-5, atol=1e-7)


# ------------------------------------------------------- Sec. 3 identities

@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_endpoint_identity_eq1(dtype):
    # R(K(C), C', {s_start..n-1}) = K(C'), bit-exact (Eq. 1; upstream rows
    # are unchanged by construction).
    cfg, W, doc, s, new = small_workload(dtype=dtype)
    stale = oracle.prefill(cfg, W, doc)
    L = len(new)
    full = np.arange(s + L, len(doc))
    rep = oracle.repair(cfg, W, stale, new, s, full)
    fresh = oracle.prefill(cfg, W, oracle.apply_edit(doc, s, new))
    assert np.array_equal(rep.k, fresh.k)
    assert np.array_equal(rep.v, fresh.v)
    assert not np.array_equal(stale.k, fresh.k)


def test_endpoint_identity_tiny_full_suffix(tiny):
    s, new = tiny["edit_start"], tiny["new_tokens"]
    n = len(tiny["doc"])
    assert n - (s + len(new)) == 308  # K = 308 is the full suffix
    rep = oracle.repair(tiny["cfg"], tiny["W"], tiny["stale"], new, s,
                        oracle.pool(n, s, len(new)))
    fresh = oracle.prefill(tiny["cfg"], tiny["W"], oracle.apply_edit(tiny["doc"], s, new))
    assert np.array_equal(rep.k, fresh.k) and np.array_equal(rep.v, fresh.v)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_noop_edit_k0_bit_identical(dtype):
    cfg, W, doc, s, new = small_workload(dtype=dtype)
    stale = oracle.prefill(cfg, W, doc)
    rep = oracle.repair(cfg, W, stale, doc[s:s + 4], s, [])
    assert np.array_equal(rep.k, stale.k) and np.array_equal(rep.v, stale.v)


def test_upstream_invariance(tiny):
    # Positions before the span cannot depend on the edit (Sec. 3).
    s, new = tiny["edit_start"], tiny["new_tokens"]
    fresh = oracle.prefill(tiny["cfg"], tiny["W"], oracle.apply_edit(tiny["doc"], s, new))
    assert np.array_equal(fresh.k[:, :s], tiny["stale"].k[:, :s])
    assert np.array_equal(fresh.v[:, :s], tiny["stale"].v[:, :s])
    assert not np.array_equal(fresh.k[:, s], tiny["stale"].k[:, s])


def test_rows_outside_P_untouched(tiny):
    s, new = tiny["edit_start"], tiny["new_tokens"]
    A = np.array([210, 250, 251, 400])
    rep = oracle.repair(tiny["cfg"], tiny["W"], tiny["stale"], new, s, A)
    P = oracle.repaired_set(s, len(new), A)
    mask = np.ones(len(tiny["doc"]), bool)
    mask[P] = False
    assert np.array_equal(rep.k[:, mask], tiny["stale"].k[:, mask])
    assert np.array_equal(rep.v[:, mask], tiny["stale"].v[:, mask])
    assert not np.array_equal(rep.k[:, P], tiny["stale"].k[:, P])


@pytest.mark.parametrize("A", [np.arange(64, 96), np.array([64, 70, 71, 100, 159])])
def test_token_major_equals_layer_major(A):
    cfg, W, doc, s, new = small_workload()
    stale = oracle.prefill(cfg, W, doc)
    lm = oracle.repair(cfg, W, stale, new, s, A)
    tm = oracle.repair(cfg, W, stale, new, s, A, token_major=True)
    assert np.array_equal(lm.k, tm.k) and np.array_equal(lm.v, tm.v)


def test_split_call_and_idempotence(tiny):
    cfg, W, s, new = tiny["cfg"], tiny["W"], tiny["edit_start"], tiny["new_tokens"]
    A = np.arange(204, 236)
    one = oracle.repair(cfg, W, tiny["stale"], new, s, A)
    first = oracle.repair(cfg, W, tiny["stale"], new, s, [])
    two = oracle.repair(cfg, W, first, new[:0], s + len(new), A)
    assert np.array_equal(one.k, two.k) and np.array_equal(one.v, two.v)
    again = oracle.repair(cfg, W, one, new, s, A)
    assert np.array_equal(one.k, again.k) and np.array_equal(one.v, again.v)


def test_repair_matches_textbook_on_repaired_rows():
    # With P the full suffix the repaired rows are the textbook forward of C'.
    cfg, W, doc, s, new = small_workload()
    stale = oracle.prefill(cfg, W, doc)
    rep = oracle.repair(cfg, W, stale, new, s, np.arange(s + 4, len(doc)))
    ref = textbook.forward(cfg, W, oracle.apply_edit(doc, s, new), want_logits=False)
    for l in range(cfg["n_layers"]):
        k = ref["layers"][l]["k"].numpy()
        np.testing.assert_allclose(rep.k[l], k, rtol=0, atol=1e-6 * np.abs(k).max())


# ---------------------------------------------------------------- selectors

def test_editlocal_golden(tiny):
    g = read_golden("editlocal_tiny.txt")
    got = oracle.select(tiny["cfg"], tiny["W"], tiny["stale"], "editlocal",
                        int(g["K"][0]), int(g["edit_start"][0]), tiny["new_tokens"])
    assert got.tolist() == [int(x) for x in g["positions"]]


def test_structural_golden():
    g = read_golden("structural_example.txt")
    n, delim = int(g["n"][0]), int(g["delim_id"][0])
    toks = np.full(n, 5, np.int32)
    toks[[int(x) for x in g["delims"]]] = delim
    cfg = synth.preset("tiny")
    cache = oracle.empty_cache(cfg, n)
    cache.tokens[:] = toks
    s, L = int(g["edit_start"][0]), int(g["edit_len"][0])
    new = toks[s:s + L]
    assert oracle.select(cfg, None, cache, "structural", 3, s, new).tolist() == \
        [int(x) for x in g["K3"]]
    assert oracle.select(cfg, None, cache, "structural", 10, s, new).tolist() == \
        [int(x) for x in g["K10"]]


def test_topk_golden():
    g = read_golden("topk_ties.txt")
    sc = np.array([float(x) for x in g["scores"]])
    for K in (4, 6, 9):
        assert oracle.topk(sc, np.arange(10), K).tolist() == [int(x) for x in g[f"K{K}"]]


def test_random_selector_properties():
    cfg = synth.preset("tiny")
    n, s, L, K = 300, 100, 4, 32
    cache = oracle.empty_cache(cfg, n)
    counts = np.zeros(n, np.int64)
    seeds = range(400)
    for seed in seeds:
        a = oracle.select(cfg, None, cache, "random", K, s, np.zeros(L, np.int32), seed)
        assert len(a) == K and len(set(a.tolist())) == K
        assert a.min() >= s + L and a.max() < n and np.all(np.diff(a) > 0)
        counts[a] += 1
    # chi-square uniformity over the pool
    pool = counts[s + L:]
    expected = len(seeds) * K / pool.size
    chi2 = float(((pool - expected) ** 2 / expected).sum())
    from scipy.stats import chi2 as chi2d
    assert chi2d.sf(chi2, pool.size - 1) > 1e-3
    # deterministic per seed, different across seeds
    a0 = oracle.select(cfg, None, cache, "random", K, s, np.zeros(L, np.int32), 0)
    a1 = oracle.select(cfg, None, cache, "random", K, s, np.zeros(L, np.int32), 1)
    assert np.array_equal(a0, oracle.select(cfg, None, cache, "random", K, s,
                                            np.zeros(L, np.int32), 0))
    assert not np.array_equal(a0, a1)


def _textbook_attention_scores(cfg, W, doc, s, new):
    """Attention-selector reading computed from two textbook forwards: the
    fresh span queries of C' and the stale keys of C, softmax over the pool,
    summed over layers, heads and span rows."""
    edited = oracle.apply_edit(doc, s, new)
    old = textbook.forward(cfg, W, doc, want_logits=False)["layers"]
    fresh = textbook.forward(cfg, W, edited, want_logits=False)["layers"]
    grp = cfg["n_heads"] // cfg["n_kv_heads"]
    e = s + len(new)
    tot = torch.zeros(len(doc), dtype=torch.float64)
    for l in range(cfg["n_layers"]):
        q = fresh[l]["q"][s:e]                                  # [S, H, dh]
        k = old[l]["k"][e:].repeat_interleave(grp, dim=1)       # [D, H, dh]
        lg = torch.einsum("shd,jhd->shj", q, k) / cfg["head_dim"] ** 0.5
        tot[e:] += torch.softmax(lg, dim=-1).sum(dim=(0, 1))
    return tot.numpy()


def test_attention_scores_match_textbook():
    cfg, W, doc, s, new = small_workload()
    stale = oracle.prefill(cfg, W, doc)
    sc, D = oracle.scores(cfg, W, stale, "attention", s, new)
    ref = _textbook_attention_scores(cfg, W, doc, s, new)
    np.testing.assert_allclose(sc, ref, rtol=0, atol=1e-6 * np.abs(ref).max())
    # probabilities over the pool sum to one per (layer, head, span row)
    total = cfg["n_layers"] * cfg["n_heads"] * len(new)
    assert abs(sc[D].sum() - total) < 1e-9 * total


def test_attention_zero_wq_gives_editlocal():
    cfg, W, doc, s, new = small_workload()
    for ly in W["layers"]:
        ly["wq"] = np.zeros_like(ly["wq"])
    stale = oracle.prefill(cfg, W, doc)
    sc, D = oracle.scores(cfg, W, stale, "attention", s, new)
    assert np.all(sc[D] == sc[D[0]])
    a = oracle.select(cfg, W, stale, "attention", 16, s, new)
    assert a.tolist() == list(range(s + 4, s + 20))


def test_cacheblend_matches_textbook():
    cfg, W, doc, s, new = small_workload()
    stale = oracle.prefill(cfg, W, doc)
    sc, D = oracle.scores(cfg, W, stale, "cacheblend", s, new)
    old = textbook.forward(cfg, W, doc, want_logits=False)["layers"][1]
    fresh = textbook.forward(cfg, W, oracle.apply_edit(doc, s, new),
                             want_logits=False)["layers"][1]
    e = s + 4
    dk = torch.linalg.vector_norm((fresh["k"] - old["k"])[e:].reshape(len(D), -1), dim=1)
    dv = torch.linalg.vector_norm((fresh["v"] - old["v"])[e:].reshape(len(D), -1), dim=1)
    ref = (dk + dv).numpy()
    np.testing.assert_allclose(sc[D], ref, rtol=0, atol=1e-5 * np.abs(ref).max())
    assert np.all(sc[D] > 0)


def test_cacheblend_equals_full_repair_deviation(tiny):
    # Layer-1 k, v of a full-suffix repair are the fresh values the score
    # compares against (same operator R); deviation is then exact.
    cfg, W, s, new = tiny["cfg"], tiny["W"], tiny["edit_start"], tiny["new_tokens"]
    n = len(tiny["doc"])
    sc, D = oracle.scores(cfg, W, tiny["stale"], "cacheblend", s, new)
    rep = oracle.repair(cfg, W, tiny["stale"], new, s, oracle.pool(n, s, len(new)))
    dk = np.sqrt(((rep.k[1, D].astype(np.float64) - tiny["stale"].k[1, D]) ** 2)
                 .reshape(len(D), -1).sum(1))
    dv = np.sqrt(((rep.v[1, D].astype(np.float64) - tiny["stale"].v[1, D]) ** 2)
                 .reshape(len(D), -1).sum(1))
    np.testing.assert_allclose(sc[D], dk + dv, rtol=1e-12, atol=0)


def test_cacheblend_unchanged_tokens_all_zero():
    cfg, W, doc, s, new = small_workload()
    stale = oracle.prefill(cfg, W, doc)
    sc, D = oracle.scores(cfg, W, stale, "cacheblend", s, doc[s:s + 4])
    assert np.all(sc == 0.0)
    assert oracle.select(cfg, W, stale, "cacheblend", 8, s, doc[s:s + 4]).tolist() == \
        list(range(s + 4, s + 12))


# ------------------------------------------------------------- NEXT rows

def test_editlocal_boundary_golden():
    g = read_golden("editlocal_boundary_example.txt")
    n, delim = int(g["n"][0]), int(g["delim_id"][0])
    toks = np.full(n, 5, np.int32)
    toks[[int(x) for x in g["delims"]]] = delim
    cfg = synth.preset("tiny")
    cache = oracle.empty_cache(cfg, n)
    cache.tokens[:] = toks
    for key in ("S13_2_K10", "S13_2_K4", "S34_2_K10", "S22_2_K16"):
        s, L, K = key.split("_")
        s, L, K = int(s[1:]), int(L), int(K[1:])
        got = oracle.select(cfg, None, cache, "editlocal_boundary", K, s, toks[s:s + L])
        assert got.tolist() == [int(x) for x in g[key]], key


def test_transplant_identity_and_noop():
    cfg, W, doc, s, new = small_workload(n=96, s=40)
    stale = oracle.prefill(cfg, W, doc)
    fresh = oracle.prefill(cfg, W, oracle.apply_edit(doc, s, new))
    full = oracle.transplant(stale, fresh, np.arange(len(doc)))
    assert np.array_equal(full.k, fresh.k) and np.array_equal(full.tokens, fresh.tokens)
    none = oracle.transplant(stale, fresh, np.array([], np.int64))
    assert np.array_equal(none.k, stale.k) and np.array_equal(none.tokens, stale.tokens)


def test_answer_logprob_matches_textbook_and_mr_endpoints():
    cfg, W, doc, s, new = small_workload(n=96, s=40)
    prompt = synth.fill_tokens(31, 3, cfg["vocab"], cfg["delim_id"])
    a_new = synth.fill_tokens(32, 2, cfg["vocab"], cfg["delim_id"])
    a_old = synth.fill_tokens(33, 2, cfg["vocab"], cfg["delim_id"])
    stale = oracle.prefill(cfg, W, doc)
    got = oracle.answer_logprob(cfg, W, stale, prompt, a_new)
    seq = np.concatenate([doc, prompt, a_new[:-1]])
    lg = textbook.forward(cfg, W, seq)["logits"][len(doc) + len(prompt) - 1:]
    ref = float(torch.log_softmax(lg, dim=-1)[torch.arange(len(a_new)),
                                              torch.as_tensor(a_new, dtype=torch.long)].mean())
    assert abs(got - ref) <= 1e-6 * abs(ref)
    # MR endpoints (Eq. 2): the oracle cache recovers 1, the stale cache 0
    fresh = oracle.prefill(cfg, W, oracle.apply_edit(doc, s, new))
    rep = oracle.repair(cfg, W, stale, new, s, oracle.pool(len(doc), s, len(new)))
    m_st = oracle.margin(cfg, W, stale, prompt, a_new, a_old)
    m_or = oracle.margin(cfg, W, fresh, prompt, a_new, a_old)
    m_rep = oracle.margin(cfg, W, rep, prompt, a_new, a_old)
    assert m_st != m_or
    assert oracle.margin_recovery(m_rep, m_st, m_or) == pytest.approx(1.0, abs=1e-12)
    assert oracle.margin_recovery(m_st, m_st, m_or) == 0.0
