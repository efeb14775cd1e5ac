"""Kernel-level check of the library's GEMMs (tcgen05/TMA for bf16 shapes)
through kvr_linear, against a float64 matmul of the same bf16 operands read
back from the device."""
import numpy as np
import pytest

from paper_2609_17983_gb300 import synth

try:
    from paper_2609_17983_gb300 import kvrepair as kv
except ImportError as _e:  # pragma: no cover
    kv, _IMPORT_ERROR = None, _e

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def model():
    if kv is None:
        raise _IMPORT_ERROR
    cfg = synth.preset("llama8b", n_layers=1)
    m = kv.Model(cfg, None, seed=0, max_context=512, max_rows=512)
    yield m
    m.close()


def f64(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


def rel(a, b):
    return float(np.abs(a - b).max() / np.abs(b).max())


@pytest.mark.parametrize("M", [1, 40, 200, 300])
def test_projections_match_fp64_matmul(model, M):
    cfg = model.cfg
    d, F = cfg["d_model"], cfg["ffn"]
    x = synth.tensor(100 + M, 5, (M, d), "bf16", std=1.0)
    xf = f64(x)
    wqkv = np.concatenate([model.read_tensor(n, 0) for n in ("wq", "wk", "wv")])
    got = kv.kvr_linear(model.h, "wqkv", 0, x, wqkv.shape[0])
    assert rel(got, xf @ f64(wqkv).T) <= 1e-3
    wo = model.read_tensor("wo", 0)
    got = kv.kvr_linear(model.h, "wo", 0, x, d)
    assert rel(got, xf @ f64(wo).T) <= 1e-3
    xd = synth.tensor(200 + M, 5, (M, F), "bf16", std=1.0)
    wd = model.read_tensor("wd", 0)
    got = kv.kvr_linear(model.h, "wd", 0, xd, d)
    assert rel(got, f64(xd) @ f64(wd).T) <= 1e-3
    g = xf @ f64(model.read_tensor("wg", 0)).T
    u = xf @ f64(model.read_tensor("wu", 0)).T
    ref = g / (1.0 + np.exp(-g)) * u
    got = kv.kvr_linear(model.h, "wgu", 0, x, F)
    assert rel(got, ref) <= 1e-2  # output rounded to bf16


def test_lm_head_matches_fp64_matmul(model):
    d = model.cfg["d_model"]
    x = synth.tensor(7, 5, (3, d), "bf16", std=1.0)
    lm = model.read_tensor("lm_head")
    got = kv.kvr_linear(model.h, "lm_head", 0, x, lm.shape[0])
    assert rel(got, f64(x) @ f64(lm).T) <= 1e-3


@pytest.mark.parametrize("M", [512, 904, 4096])
def test_many_row_projections_match_fp64_matmul(M):
    # a prefill chunk's row counts: the grouped data-parallel tiling (whole
    # tiles per CTA, token tiles of up to 256 rows with a ragged last one;
    # at 904 rows gate/up's 224 feature tiles in 38 groups of 5 or 6); the
    # fp64 reference on a sample of rows from every token tile
    cfg = synth.preset("llama8b", n_layers=1)
    m = kv.Model(cfg, None, seed=0, max_context=512, max_rows=4096)
    d, F = cfg["d_model"], cfg["ffn"]
    rows = np.unique(np.concatenate([np.arange(0, M, 61), np.arange(M - 8, M)]))
    x = synth.tensor(300 + M, 5, (M, d), "bf16", std=1.0)
    xf = f64(x[rows])
    for name, w in (("wqkv", np.concatenate([m.read_tensor(n, 0) for n in ("wq", "wk", "wv")])),
                    ("wo", m.read_tensor("wo", 0))):
        got = kv.kvr_linear(m.h, name, 0, x, w.shape[0])
        assert rel(got[rows], xf @ f64(w).T) <= 1e-3, name
    xd = synth.tensor(400 + M, 5, (M, F), "bf16", std=1.0)
    wd = m.read_tensor("wd", 0)
    got = kv.kvr_linear(m.h, "wd", 0, xd, d)
    assert rel(got[rows], f64(xd[rows]) @ f64(wd).T) <= 1e-3
    g = xf @ f64(m.read_tensor("wg", 0)).T
    u = xf @ f64(m.read_tensor("wu", 0)).T
    got = kv.kvr_linear(m.h, "wgu", 0, x, F)
    assert rel(got[rows], g / (1.0 + np.exp(-g)) * u) <= 1e-2  # output rounded to bf16
    m.close()
