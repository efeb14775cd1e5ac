"""Seeded synthetic inputs: model presets, random-init weights, documents, edits.

This module generates inputs only; it holds none of the repair method's
arithmetic.  Tests and the benchmark hand its outputs both to the CUDA library
and to the CPU oracle.  It imports neither of them.

Weights follow one counter-based definition, which the CUDA library also
implements on the device (``kvr_model_create`` with no weights):

* SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014): ``out(s, i) = mix(s + (i + 1) * GAMMA)`` is the
  i-th output of a generator seeded with s, where mix is the published
  two-round xor-shift-multiply finaliser.
* Tensor t of model seed S draws from the stream ``s_t = out(S, t)``; element
  i (row-major, ``[out_features][in_features]``) is ``r = out(s_t, i)``.
* The value is approximately N(0, std): the four 16-bit lanes of r are summed
  (Irwin-Hall with n = 4; exact mean 2 * 65535 and variance (65536^2 - 1) / 3),
  centred, and scaled in double by ``c = std / sqrt((65536^2 - 1) / 3)``; the
  product is rounded to fp32 (nearest even) and, for bf16 models, on to bf16
  (nearest even).  Every step is exact or correctly rounded, so the host and
  device produce identical bits.
* RMSNorm gains are 1.

The paper evaluates trained Llama-3.1-8B, Qwen3-8B and Mistral-7B on HotpotQA
backgrounds; neither the weights nor the data are available here, so the
presets below are random-init models of those shapes and documents are uniform
random token ids (the delimiter id excluded from the fill).
"""
from __future__ import annotations

import math
import os

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
LANE_MEAN_SUM = 2 * 65535          # mean of the sum of four 16-bit lanes
WEIGHT_STD = 0.02

# ------------------------------------------------------------------ presets

PRESETS = {
    # Tiny Llama-style decoder, fp32 (the small workload the oracle finishes in seconds).
    "tiny": dict(vocab=1024, d_model=256, n_layers=2, n_heads=4, n_kv_heads=2,
                 head_dim=64, ffn=688, rope_theta=10000.0, rms_eps=1e-5,
                 qkv_bias=False, dtype="fp32", delim_id=13),
    # Llama-3-8B shape, bf16.
    "llama8b": dict(vocab=128256, d_model=4096, n_layers=32, n_heads=32, n_kv_heads=8,
                    head_dim=128, ffn=14336, rope_theta=500000.0, rms_eps=1e-5,
                    qkv_bias=False, dtype="bf16", delim_id=13),
    # Qwen2.5-7B shape (QKV bias), bf16.
    "qwen7b": dict(vocab=152064, d_model=3584, n_layers=28, n_heads=28, n_kv_heads=4,
                   head_dim=128, ffn=18944, rope_theta=1000000.0, rms_eps=1e-6,
                   qkv_bias=True, dtype="bf16", delim_id=13),
    # Mistral-7B shape, bf16.
    "mistral7b": dict(vocab=32768, d_model=4096, n_layers=32, n_heads=32, n_kv_heads=8,
                      head_dim=128, ffn=14336, rope_theta=1000000.0, rms_eps=1e-5,
                      qkv_bias=False, dtype="bf16", delim_id=13),
}


def preset(name: str, **overrides) -> dict:
    cfg = dict(PRESETS[name])
    cfg.update(overrides)
    return cfg


# Tensor ids of the weight streams.  Layer l uses LAYER_BASE + LAYER_STRIDE*l + k.
TID_EMBED, TID_LM_HEAD = 0, 1
LAYER_BASE, LAYER_STRIDE = 8, 16
LAYER_TIDS = dict(wq=0, wk=1, wv=2, wo=3, wg=4, wu=5, wd=6, bq=7, bk=8, bv=9)


def layer_tid(layer: int, name: str) -> int:
    return LAYER_BASE + LAYER_STRIDE * layer + LAYER_TIDS[name]


# --------------------------------------------------------------- SplitMix64

def mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 finaliser (two xor-shift-multiply rounds and a final xor-shift)."""
    z = np.asarray(z, np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def stream_out(seed, idx) -> np.ndarray:
    """out(seed, i) = mix(seed + (i + 1) * GAMMA), the i-th SplitMix64 output."""
    seed = np.uint64(int(seed) & 0xFFFFFFFFFFFFFFFF)
    idx = np.asarray(idx, np.uint64)
    with np.errstate(over="ignore"):
        return mix64(seed + (idx + np.uint64(1)) * GAMMA)


def tensor_seed(model_seed: int, tid: int) -> int:
    return int(stream_out(model_seed, np.array([tid], np.uint64))[0])


def weight_scale(std: float = WEIGHT_STD) -> float:
    return std / math.sqrt((65536.0 * 65536.0 - 1.0) / 3.0)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns, round to nearest even (inputs are finite)."""
    u = np.ascontiguousarray(x, np.float32).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_values(model_seed: int, tid: int, idx: np.ndarray, dtype: str,
                  std: float = WEIGHT_STD) -> np.ndarray:
    """Weight values at element indices idx of tensor tid (see module doc)."""
    r = stream_out(tensor_seed(model_seed, tid), idx)
    return _lanes_to_values(r, dtype, std)


def _lanes_to_values(r: np.ndarray, dtype: str, std: float) -> np.ndarray:
    """Irwin-Hall(4) of the 16-bit lanes of r, centred, scaled, rounded (in place on r)."""
    m16 = np.uint64(0xFFFF)
    t = np.empty_like(r)
    s = np.bitwise_and(r, m16)
    for sh in (16, 32):
        np.right_shift(r, np.uint64(sh), out=t)
        np.bitwise_and(t, m16, out=t)
        s += t
    np.right_shift(r, np.uint64(48), out=t)
    s += t
    x = s.view(np.int64)
    x -= LANE_MEAN_SUM
    f = (x.astype(np.float64) * weight_scale(std)).astype(np.float32)
    return f32_to_bf16_bits(f) if dtype == "bf16" else f


def _contiguous_values(tseed: int, start: int, count: int, dtype: str, std: float) -> np.ndarray:
    """Values of elements start..start+count-1 of the stream tseed."""
    z = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    t = np.empty_like(z)
    with np.errstate(over="ignore"):
        z *= GAMMA
        z += np.uint64(tseed)
        np.right_shift(z, np.uint64(30), out=t)
        z ^= t
        z *= _M1
        np.right_shift(z, np.uint64(27), out=t)
        z ^= t
        z *= _M2
        np.right_shift(z, np.uint64(31), out=t)
        z ^= t
    return _lanes_to_values(z, dtype, std)


def tensor(model_seed: int, tid: int, shape, dtype: str, std: float = WEIGHT_STD,
           chunk: int = 1 << 21) -> np.ndarray:
    n = int(np.prod(shape))
    out = np.empty(n, np.uint16 if dtype == "bf16" else np.float32)
    tseed = tensor_seed(model_seed, tid)

    def fill(b):
        e = min(n, b + chunk)
        out[b:e] = _contiguous_values(tseed, b, e - b, dtype, std)

    starts = range(0, n, chunk)
    if n > 4 * chunk:
        from concurrent.futures import ThreadPoolExecutor
        with ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
            list(ex.map(fill, starts))
    else:
        for b in starts:
            fill(b)
    return out.reshape(shape)


def rows(model_seed: int, tid: int, row_ids, ncols: int, dtype: str) -> np.ndarray:
    """Selected rows of a [*, ncols] tensor (e.g. embedding rows of some tokens)."""
    row_ids = np.asarray(row_ids, np.uint64)
    idx = (row_ids[:, None] * np.uint64(ncols) + np.arange(ncols, dtype=np.uint64)[None, :])
    return normal_values(model_seed, tid, idx.reshape(-1), dtype).reshape(len(row_ids), ncols)


def ones(n: int, dtype: str) -> np.ndarray:
    return np.full(n, 0x3F80, np.uint16) if dtype == "bf16" else np.ones(n, np.float32)


def layer_weights(cfg: dict, model_seed: int, layer: int) -> dict:
    d, H, G, dh, F, dt = (cfg["d_model"], cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"],
                          cfg["ffn"], cfg["dtype"])
    t = lambda name, shape: tensor(model_seed, layer_tid(layer, name), shape, dt)
    ly = dict(attn_norm=ones(d, dt), mlp_norm=ones(d, dt),
              wq=t("wq", (H * dh, d)), wk=t("wk", (G * dh, d)), wv=t("wv", (G * dh, d)),
              wo=t("wo", (d, H * dh)), wg=t("wg", (F, d)), wu=t("wu", (F, d)),
              wd=t("wd", (d, F)))
    if cfg.get("qkv_bias"):
        ly.update(bq=t("bq", (H * dh,)), bk=t("bk", (G * dh,)), bv=t("bv", (G * dh,)))
    return ly


def weights(cfg: dict, model_seed: int = 0, n_layers: int | None = None,
            embed: bool = True, lm_head: bool = True) -> dict:
    """Canonical host weights {embed, final_norm, lm_head, layers: [...]}: fp32
    arrays for fp32 models, uint16 bf16 bit patterns for bf16 models."""
    L = cfg["n_layers"] if n_layers is None else n_layers
    d, V, dt = cfg["d_model"], cfg["vocab"], cfg["dtype"]
    return dict(
        embed=tensor(model_seed, TID_EMBED, (V, d), dt) if embed else None,
        lm_head=tensor(model_seed, TID_LM_HEAD, (V, d), dt) if lm_head else None,
        final_norm=ones(d, dt),
        layers=[layer_weights(cfg, model_seed, l) for l in range(L)])


# ------------------------------------------------------- stale KV caches

# Spread of the synthetic cache entries: a K or V entry of these models is a
# projection of an RMS-normalised row (unit RMS) by N(0, 0.02^2) weights over
# d_model = 4096 inputs, whose standard deviation is 0.02 * sqrt(4096) = 1.28.
KV_STD = 1.28
TID_CACHE_K, TID_CACHE_V = 1001, 1002


def kv_rows(seed: int, n: int, n_layers: int, n_kv_heads: int, head_dim: int, dtype: str,
            std: float = KV_STD) -> tuple[np.ndarray, np.ndarray]:
    """A seeded synthetic stale cache: K and V rows [n][n_layers][n_kv_heads][head_dim]
    with entries approximately N(0, std^2), from the weight generator's counter-based
    streams (tensor ids TID_CACHE_K / TID_CACHE_V of `seed`); bf16 bit patterns for
    bf16, else float32.  Used where a test or a timing needs a cached state K(C)
    of a long context that no CPU prefill could produce: repair is defined over
    any stale cache."""
    shape = (n, n_layers, n_kv_heads, head_dim)
    return (tensor(seed, TID_CACHE_K, shape, dtype, std),
            tensor(seed, TID_CACHE_V, shape, dtype, std))


# --------------------------------------------------------- documents, edits

def _uniform_ints(seed: int, count: int, lo: int, hi: int) -> np.ndarray:
    """count integers uniform in [lo, hi) from stream `seed` (modulo reduction)."""
    r = stream_out(seed, np.arange(count, dtype=np.uint64))
    return (lo + (r % np.uint64(hi - lo)).astype(np.int64)).astype(np.int64)


def fill_tokens(seed: int, count: int, vocab: int, delim_id: int) -> np.ndarray:
    """Uniform token ids from [0, vocab) without the delimiter id."""
    t = _uniform_ints(seed, count, 0, vocab - 1)
    t = t + (t >= delim_id)
    return t.astype(np.int32)


def document(seed: int, n: int, vocab: int, delim_id: int = 13,
             delim_gap: tuple[int, int] | None = None) -> np.ndarray:
    """A document of n uniform random token ids; if delim_gap=(lo, hi), the
    delimiter id is placed after every U[lo, hi] tokens (seeded)."""
    doc = fill_tokens(seed, n, vocab, delim_id)
    if delim_gap is not None:
        lo, hi = delim_gap
        gaps = _uniform_ints(int(stream_out(seed, np.array([1 << 40], np.uint64))[0]),
                             n // lo + 2, lo, hi + 1)
        p = -1
        for g in gaps:
            p += int(g) + 1
            if p >= n:
                break
            doc[p] = delim_id
    return doc


def edit_tokens(seed: int, old: np.ndarray, vocab: int, delim_id: int = 13) -> np.ndarray:
    """New ids for an edit span, each different from the id it replaces."""
    old = np.asarray(old, np.int32)
    new = fill_tokens(seed, old.shape[0], vocab, delim_id)
    same = new == old
    # shift colliding ids to the next non-delimiter id
    new[same] = (new[same] + 1) % vocab
    new[new == delim_id] = (new[new == delim_id] + 1) % vocab
    return new.astype(np.int32)


def seeded_int(seed: int, lo: int, hi: int) -> int:
    """One integer uniform in [lo, hi] from stream `seed`."""
    return int(_uniform_ints(seed, 1, lo, hi + 1)[0])


def batch_edits(seed: int, n: int, n_edits: int, span: tuple[int, int], K: int,
                margin: int = 64) -> list[tuple[int, int]]:
    """n_edits non-overlapping (start, length) edits in one document of length
    n, spans U[span], each followed by room for a K-position window."""
    rng_lens = _uniform_ints(seed, n_edits, span[0], span[1] + 1)
    slot = (n - margin) // n_edits
    out = []
    for e in range(n_edits):
        length = int(rng_lens[e])
        lo = e * slot + margin // 2
        hi = lo + slot - length - K - margin // 2
        start = seeded_int(seed * 131 + e + 1, lo, max(lo, hi))
        out.append((start, length))
    return out


# ------------------------------------------------------------ the workloads

def workload(name: str) -> dict:
    """The seeded synthetic workloads.  Returns a dict with the model preset,
    the cached document, the edit and the budgets."""
    if name == "tiny":
        cfg = preset("tiny")
        doc = document(1, 512, cfg["vocab"], cfg["delim_id"])
        s, L = 200, 4
        new = edit_tokens(2, doc[s:s + L], cfg["vocab"], cfg["delim_id"])
        return dict(cfg=cfg, doc=doc, edit_start=s, new_tokens=new, K=32, Ks=(0, 32, 308))
    if name == "llama8b":
        cfg = preset("llama8b")
        doc = document(1, 5000, cfg["vocab"], cfg["delim_id"])
        s, L = 2500, 8
        new = edit_tokens(2, doc[s:s + L], cfg["vocab"], cfg["delim_id"])
        return dict(cfg=cfg, doc=doc, edit_start=s, new_tokens=new, K=32, Ks=(32,))
    if name == "qwen7b":
        cfg = preset("qwen7b")
        doc = document(1, 5000, cfg["vocab"], cfg["delim_id"])
        s, L = seeded_int(3, 1000, 4000), 6
        new = edit_tokens(2, doc[s:s + L], cfg["vocab"], cfg["delim_id"])
        return dict(cfg=cfg, doc=doc, edit_start=s, new_tokens=new, K=32,
                    Ks=(8, 16, 32, 64, 128))
    if name == "mistral7b":
        cfg = preset("mistral7b")
        doc = document(1, 5000, cfg["vocab"], cfg["delim_id"], delim_gap=(40, 80))
        s, L = seeded_int(4, 1000, 4000), 10
        new = edit_tokens(2, doc[s:s + L], cfg["vocab"], cfg["delim_id"])
        return dict(cfg=cfg, doc=doc, edit_start=s, new_tokens=new, K=32, Ks=(32,))
    raise ValueError(f"unknown workload {name!r}")
