"""Plain CPU oracle for budgeted KV-cache repair.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` import this package.  It shares no code with
the CUDA library (``paper_2609_17983_gb300``) and imports nothing from it; the
two meet only in the seeded inputs the tests hand to both.

The model forward, the repair operator and the two model-based selectors live
in ``kvr_oracle.c`` (IEEE double, deterministic, see its header).  This module
loads it through ctypes (compiling it with gcc on first use), and implements
in Python the parts that are closed-form: the candidate pool, the three
text/position selectors of Table 1 and the top-K rule.

Paper: "Contiguity, Not Importance: Budgeted Repair of Stale KV Caches After
Document Edits".  Sec. 3 defines the repair interface (operator R, Eq. 1), the
pool D and the selection policies (Table 1).

Pin status (what each function is checked against, in tests/test_oracle_*.py):
  prefill / recompute  -- textbook decoder composed from torch library calls in
                          fp64 (scaled_dot_product_attention, rms_norm, a
                          complex-number RoPE), Eq. 1 endpoint identity,
                          no-op edit, token-major brute force, upstream
                          invariance, split-call and idempotence.
  bf16 path            -- the same textbook decoder with the bf16 path's
                          rounding points (torch's own bf16 conversions, an
                          attention written out over all heads), to 1e-9;
                          the Eq. 1 identities hold bit-exact on it too.
  logits               -- the same textbook decoder run over C' + query.
  editlocal/structural -- closed forms and hand-written golden cases.
  editlocal_boundary   -- hand-written golden case.
  logits_all / answer_logprob -- the textbook decoder run over C' + query.
  transplant           -- identity (all positions) and no-op (none) cases.
  random               -- published SplitMix64 test vectors, uniformity.
  attention score      -- the reading computed from two textbook forwards (the
                          fresh span queries of C', the stale pool keys of C,
                          softmax over the pool, summed over layers, heads and
                          span rows); zero W_q gives uniform scores (ties ->
                          EditLocal set); the scores sum to layers*heads*|S|.
  cacheblend score     -- the layer-1 K/V deviation between two textbook
                          forwards (C' and C) over the pool; equal to the
                          deviation a full-suffix repair leaves; an edit that
                          changes no token gives all-zero deviation.
  topk                 -- hand-written golden cases with ties and NaN.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kvr_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

GOLDEN = 0x9E3779B97F4A7C15
MASK64 = (1 << 64) - 1


def build(force: bool = False) -> str:
    """Compile kvr_oracle.c into _build/liboracle.so (OpenMP if available)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
            "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Config(ctypes.Structure):
    _fields_ = [("vocab", ctypes.c_int32), ("d_model", ctypes.c_int32),
                ("n_layers", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("ffn", ctypes.c_int32), ("qkv_bias", ctypes.c_int32),
                ("wdtype", ctypes.c_int32), ("cdtype", ctypes.c_int32),
                ("operands", ctypes.c_int32),
                ("rope_theta", ctypes.c_double), ("rms_eps", ctypes.c_double)]


_PP = ctypes.POINTER(ctypes.c_void_p)


class _Weights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("lm_head", ctypes.c_void_p),
                ("attn_norm", _PP), ("wq", _PP), ("wk", _PP), ("wv", _PP), ("wo", _PP),
                ("bq", _PP), ("bk", _PP), ("bv", _PP),
                ("mlp_norm", _PP), ("wg", _PP), ("wu", _PP), ("wd", _PP)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            lib.orc_set_threads.argtypes = [ctypes.c_int]
            lib.orc_set_threads.restype = ctypes.c_int
            common = [ctypes.POINTER(_Config), ctypes.POINTER(_Weights), P, P, ctypes.c_int]
            lib.orc_recompute.argtypes = common + [P, P, ctypes.c_int, P]
            lib.orc_recompute_token_major.argtypes = common + [P, P, ctypes.c_int, P]
            lib.orc_score_attention.argtypes = common + [ctypes.c_int, P, ctypes.c_int,
                                                         ctypes.c_int, P]
            lib.orc_score_cacheblend.argtypes = common + [ctypes.c_int, P, ctypes.c_int,
                                                          ctypes.c_int, P]
            lib.orc_logits.argtypes = common + [ctypes.c_int, P, ctypes.c_int, P]
            lib.orc_logits_all.argtypes = common + [ctypes.c_int, P, ctypes.c_int, P]
            for f in (lib.orc_recompute, lib.orc_recompute_token_major,
                      lib.orc_score_attention, lib.orc_score_cacheblend, lib.orc_logits,
                      lib.orc_logits_all):
                f.restype = ctypes.c_int
            _lib = lib
    return _lib


def set_threads(n: int) -> int:
    """Set the OpenMP thread count (n <= 0 keeps it); returns the count in use."""
    return int(_load().orc_set_threads(int(n)))


# ----------------------------------------------------------------- marshalling

def _wdtype(cfg) -> int:
    return 1 if cfg["dtype"] == "bf16" else 0


# Operand precision of the matrix products (kvr_oracle.c, orc_config.operands):
# "fp64" keeps them in double; "bf16" rounds every operand of a matrix product
# to bf16, as the bf16 path does; "bf16_dense" only those of the weight
# products; "bf16_f32sums" is the bf16 path with the weight products' results
# and the residual stream rounded to fp32 (a null control: how far last-bit
# changes of the sums carry through the layers).  A config's "operands" key
# selects it; by default a bf16 model is computed on the bf16 path and an
# fp32 model in double.
OPERANDS = {"fp64": 0, "bf16_dense": 1, "bf16": 3, "bf16_f32sums": 7}


def _cfg_struct(cfg) -> _Config:
    bf = _wdtype(cfg)
    return _Config(cfg["vocab"], cfg["d_model"], cfg["n_layers"], cfg["n_heads"],
                   cfg["n_kv_heads"], cfg["head_dim"], cfg["ffn"],
                   1 if cfg.get("qkv_bias") else 0, bf, bf,
                   OPERANDS[cfg.get("operands", "bf16" if bf else "fp64")],
                   float(cfg["rope_theta"]), float(cfg["rms_eps"]))


class _WeightsHandle:
    """Keeps the numpy arrays and pointer tables alive for one call."""

    def __init__(self, cfg, W):
        want = np.uint16 if cfg["dtype"] == "bf16" else np.float32
        self.keep = []

        def ptr(a):
            if a is None:
                return None
            a = np.ascontiguousarray(a)
            if a.dtype != want:
                raise TypeError(f"weight dtype {a.dtype}, expected {want}")
            self.keep.append(a)
            return a.ctypes.data

        def table(key, layers):
            arr = (ctypes.c_void_p * len(layers))(*[ptr(ly.get(key)) for ly in layers])
            self.keep.append(arr)
            return ctypes.cast(arr, _PP)

        L = W["layers"]
        if len(L) < cfg["n_layers"]:
            raise ValueError("fewer layer weights than n_layers")
        self.s = _Weights(ptr(W["embed"]), ptr(W["final_norm"]), ptr(W.get("lm_head")),
                          table("attn_norm", L), table("wq", L), table("wk", L),
                          table("wv", L), table("wo", L), table("bq", L), table("bk", L),
                          table("bv", L), table("mlp_norm", L), table("wg", L),
                          table("wu", L), table("wd", L))


@dataclass
class Cache:
    """Oracle KV cache: k, v = float32 [n_layers, cap, n_kv_heads, head_dim]
    holding values of the cache dtype; tokens = int32[n] of the cached context."""
    k: np.ndarray
    v: np.ndarray
    tokens: np.ndarray

    @property
    def n(self) -> int:
        return int(self.tokens.shape[0])

    def copy(self, cap: int | None = None) -> "Cache":
        cap = self.k.shape[1] if cap is None else cap
        L, c0, G, dh = self.k.shape
        k = np.zeros((L, cap, G, dh), np.float32)
        v = np.zeros((L, cap, G, dh), np.float32)
        c = min(c0, cap)
        k[:, :c] = self.k[:, :c]
        v[:, :c] = self.v[:, :c]
        return Cache(k, v, self.tokens.copy())


def empty_cache(cfg, n: int, cap: int | None = None) -> Cache:
    cap = n if cap is None else cap
    shape = (cfg["n_layers"], cap, cfg["n_kv_heads"], cfg["head_dim"])
    return Cache(np.zeros(shape, np.float32), np.zeros(shape, np.float32),
                 np.zeros(n, np.int32))


def _check(rc: int, what: str):
    if rc != 0:
        raise RuntimeError(f"oracle {what} failed with code {rc}")


def recompute(cfg, W, cache: Cache, tokens, rows, token_major: bool = False,
              want_h: bool = False):
    """Operator R (Sec. 3): recompute rows (strictly increasing positions) of
    `cache` in place from `tokens`, layer-major (or token-major brute force).
    Returns the rows' final residual stream [m, d_model] if want_h."""
    lib = _load()
    tokens = np.ascontiguousarray(tokens, np.int32)
    rows = np.ascontiguousarray(rows, np.int64)
    m = int(rows.shape[0])
    h = np.zeros((max(m, 1), cfg["d_model"]), np.float64) if want_h else None
    wh = _WeightsHandle(cfg, W)
    c = _cfg_struct(cfg)
    fn = lib.orc_recompute_token_major if token_major else lib.orc_recompute
    _check(fn(ctypes.byref(c), ctypes.byref(wh.s), cache.k.ctypes.data, cache.v.ctypes.data,
              cache.k.shape[1], tokens.ctypes.data, rows.ctypes.data, m,
              h.ctypes.data if want_h else None), "recompute")
    return h[:m] if want_h else None


def prefill(cfg, W, tokens, cap: int | None = None) -> Cache:
    """Full prefill K(C): operator R with P = {0..n-1} on an empty cache."""
    tokens = np.ascontiguousarray(tokens, np.int32)
    n = int(tokens.shape[0])
    cache = empty_cache(cfg, n, cap)
    cache.tokens[:] = tokens
    recompute(cfg, W, cache, tokens, np.arange(n))
    return cache


def apply_edit(tokens, edit_start: int, new_tokens) -> np.ndarray:
    """C' = C with the half-open span [edit_start, edit_start + len) replaced
    (Sec. 3 "Question Setting": one contiguous, length-preserving edit)."""
    t = np.array(tokens, np.int32, copy=True)
    new_tokens = np.asarray(new_tokens, np.int32)
    e = edit_start + new_tokens.shape[0]
    if edit_start < 0 or e > t.shape[0]:
        raise ValueError("edit span outside the context")
    t[edit_start:e] = new_tokens
    return t


def repaired_set(edit_start: int, edit_len: int, positions) -> np.ndarray:
    """P = S U A with S = [s_start, s_end) and A a subset of D = [s_end, n)."""
    s_end = edit_start + edit_len
    a = np.asarray(positions, np.int64)
    if a.size and (np.any(a < s_end) or np.any(np.diff(a) <= 0)):
        raise ValueError("positions must be strictly increasing and >= edit end")
    return np.concatenate([np.arange(edit_start, s_end, dtype=np.int64), a])


def repair(cfg, W, cache: Cache, new_tokens, edit_start: int, positions,
           token_major: bool = False) -> Cache:
    """R(K(C), C', S U A) on a copy of `cache`; returns the repaired copy."""
    new_tokens = np.asarray(new_tokens, np.int32)
    out = cache.copy()
    out.tokens = apply_edit(cache.tokens, edit_start, new_tokens)
    P = repaired_set(edit_start, new_tokens.shape[0], positions)
    if P.size:
        if P[-1] >= cache.n:
            raise ValueError("position beyond the context")
        recompute(cfg, W, out, out.tokens, P, token_major=token_major)
    return out


def logits(cfg, W, cache: Cache, query) -> np.ndarray:
    """Fresh-query logits (Sec. 3): the query tokens at positions n..n+m-1
    attend to the cache; the document's entries are not modified.  Returns
    float64[vocab] for the last query row."""
    lib = _load()
    query = np.asarray(query, np.int32)
    n, m = cache.n, int(query.shape[0])
    work = cache.copy(cap=n + m)
    toks = np.concatenate([cache.tokens, query]).astype(np.int32)
    out = np.zeros(cfg["vocab"], np.float64)
    wh = _WeightsHandle(cfg, W)
    c = _cfg_struct(cfg)
    _check(lib.orc_logits(ctypes.byref(c), ctypes.byref(wh.s), work.k.ctypes.data,
                          work.v.ctypes.data, n + m, n, toks.ctypes.data, m,
                          out.ctypes.data), "logits")
    return out


def logits_all(cfg, W, cache: Cache, query) -> np.ndarray:
    """Logits [m, vocab] of every query row (positions n..n+m-1)."""
    lib = _load()
    query = np.asarray(query, np.int32)
    n, m = cache.n, int(query.shape[0])
    work = cache.copy(cap=n + m)
    toks = np.concatenate([cache.tokens, query]).astype(np.int32)
    out = np.zeros((m, cfg["vocab"]), np.float64)
    wh = _WeightsHandle(cfg, W)
    c = _cfg_struct(cfg)
    _check(lib.orc_logits_all(ctypes.byref(c), ctypes.byref(wh.s), work.k.ctypes.data,
                              work.v.ctypes.data, n + m, n, toks.ctypes.data, m,
                              out.ctypes.data), "logits_all")
    return out


def answer_logprob(cfg, W, cache: Cache, prompt, answer) -> float:
    """Length-averaged teacher-forced log-probability of `answer` after the
    cached context and `prompt` (the quantity whose a_new - a_old difference
    is the margin m_x of Eq. 2)."""
    prompt = np.asarray(prompt, np.int32)
    answer = np.asarray(answer, np.int32)
    feed = np.concatenate([prompt, answer[:-1]])
    lg = logits_all(cfg, W, cache, feed)[len(prompt) - 1:]
    mx = lg.max(axis=1, keepdims=True)
    lse = mx[:, 0] + np.log(np.exp(lg - mx).sum(axis=1))
    return float(np.mean(lg[np.arange(len(answer)), answer] - lse))


def margin(cfg, W, cache: Cache, prompt, a_new, a_old) -> float:
    """m_x (Eq. 2): answer log-probability of a_new minus that of a_old."""
    return answer_logprob(cfg, W, cache, prompt, a_new) - answer_logprob(cfg, W, cache, prompt,
                                                                          a_old)


def margin_recovery(m_repaired: float, m_stale: float, m_oracle: float) -> float:
    """MR (Eq. 2): (m_repaired - m_stale) / (m_oracle - m_stale), unclipped."""
    return (m_repaired - m_stale) / (m_oracle - m_stale)


def transplant(dst: Cache, src: Cache, positions) -> Cache:
    """Transplant (Sec. 3): a copy of dst whose K/V of every layer and token
    at `positions` come from src."""
    positions = np.asarray(positions, np.int64)
    out = dst.copy()
    out.k[:, positions] = src.k[:, positions]
    out.v[:, positions] = src.v[:, positions]
    out.tokens[positions] = src.tokens[positions]
    return out


# ------------------------------------------------------------------ selectors

POLICIES = ("editlocal", "structural", "attention", "cacheblend", "random",
            "editlocal_boundary")


def pool(n: int, edit_start: int, edit_len: int) -> np.ndarray:
    """Candidate pool D = [s_end, n).  The paper writes [s_end, n-1); the
    reading taken here includes n-1 so that K = n - s_end is the full suffix."""
    return np.arange(edit_start + edit_len, n, dtype=np.int64)


def splitmix64(state: int) -> int:
    """First output of a SplitMix64 generator (Steele, Lea & Flood 2014) whose
    state is `state`: advance the state by the golden gamma, then mix."""
    z = (state + GOLDEN) & MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


def topk(scores, eligible, K: int) -> np.ndarray:
    """Top-K of `scores` over the eligible positions: descending score, ties
    to the lowest index, NaN ranked as -inf; returned in ascending order."""
    idx = [int(j) for j in np.asarray(eligible)]

    def key(j):
        s = scores[j]
        if isinstance(s, (float, np.floating)):
            s = -np.inf if np.isnan(s) else float(s)
        return (-s, j)

    chosen = sorted(idx, key=key)[:max(K, 0)]
    return np.array(sorted(chosen), np.int64)


def scores(cfg, W, cache: Cache, policy: str, edit_start: int, new_tokens, seed: int = 0):
    """Per-position selector scores over the pool (Table 1).  Returns
    (scores, eligible) where scores is indexable by position."""
    new_tokens = np.asarray(new_tokens, np.int32)
    L = new_tokens.shape[0]
    n = cache.n
    s_end = edit_start + L
    D = pool(n, edit_start, L)
    toks = apply_edit(cache.tokens, edit_start, new_tokens)
    if policy == "editlocal":
        return {int(j): -float(j - s_end) for j in D}, D
    if policy == "structural":
        delim = cfg["delim_id"]
        elig = np.array([j for j in D if toks[j] == delim], np.int64)
        return {int(j): -float(j - s_end) for j in elig}, elig
    if policy == "random":
        return {int(j): splitmix64(seed ^ ((int(j) * GOLDEN) & MASK64)) for j in D}, D
    if policy == "editlocal_boundary":
        # Sec. 5.2: through the next document boundary (first delimiter at or
        # after the span end, inclusive; the context end if there is none)
        delim = cfg["delim_id"]
        hits = [int(j) for j in D if toks[j] == delim]
        b = hits[0] if hits else n - 1
        elig = np.arange(s_end, b + 1, dtype=np.int64)
        return {int(j): -float(j - s_end) for j in elig}, elig
    if policy in ("attention", "cacheblend"):
        lib = _load()
        work = cache.copy()
        out = np.zeros(n, np.float64)
        wh = _WeightsHandle(cfg, W)
        c = _cfg_struct(cfg)
        fn = lib.orc_score_attention if policy == "attention" else lib.orc_score_cacheblend
        if L > 0:
            _check(fn(ctypes.byref(c), ctypes.byref(wh.s), work.k.ctypes.data,
                      work.v.ctypes.data, work.k.shape[1], n, toks.ctypes.data,
                      edit_start, s_end, out.ctypes.data), policy)
        return out, D
    raise ValueError(f"unknown policy {policy!r}")


def select(cfg, W, cache: Cache, policy: str, K: int, edit_start: int, new_tokens,
           seed: int = 0) -> np.ndarray:
    """A_pi: K positions of the pool chosen by `policy`, ascending."""
    sc, elig = scores(cfg, W, cache, policy, edit_start, new_tokens, seed)
    return topk(sc, elig, K)
