"""ctypes binding of libkvrepair (argument marshalling only).

The functions below carry the names of the C entry points in
``include/kvrepair.h`` and forward to them; every step of the method runs in
the library's CUDA kernels.  Importing this module loads
``libkvrepair.so`` from this package directory (``libkvrepair_trace.so``, the
build with the device timeline trace, when ``KVR_LIB=trace``) and raises
ImportError if it has not been built (``__graft_entry__.build()``): there is
no fallback.

``Model`` and ``Cache`` are thin owners of the C handles for convenience.
"""
from __future__ import annotations

import atexit
import ctypes
import os
import weakref

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libkvrepair_trace.so" if os.environ.get("KVR_LIB") == "trace"
                        else "libkvrepair.so")
if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
_lib = ctypes.CDLL(LIB_PATH)

KVR_OK = 0
ERRORS = {1: "KVR_E_INVAL", 2: "KVR_E_RANGE", 3: "KVR_E_NOMEM", 4: "KVR_E_CUDA",
          5: "KVR_E_DEVICE_TIMEOUT", 6: "KVR_E_UNSUPPORTED", 7: "KVR_E_POISONED"}
DTYPES = {"fp32": 0, "bf16": 1}
POLICIES = {"editlocal": 0, "structural": 1, "attention": 2, "cacheblend": 3, "random": 4,
            "editlocal_boundary": 5}


class KvrError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{ERRORS.get(code, code)}: {msg}")
        self.code = code


class ModelConfig(ctypes.Structure):
    _fields_ = [("vocab", ctypes.c_int32), ("d_model", ctypes.c_int32),
                ("n_layers", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("ffn", ctypes.c_int32), ("qkv_bias", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("delim_id", ctypes.c_int32),
                ("rope_theta", ctypes.c_double), ("rms_eps", ctypes.c_double),
                ("max_context", ctypes.c_int32), ("max_rows", ctypes.c_int32)]


_PP = ctypes.POINTER(ctypes.c_void_p)


class Weights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("lm_head", ctypes.c_void_p),
                ("attn_norm", _PP), ("wq", _PP), ("wk", _PP), ("wv", _PP), ("wo", _PP),
                ("bq", _PP), ("bk", _PP), ("bv", _PP),
                ("mlp_norm", _PP), ("wg", _PP), ("wu", _PP), ("wd", _PP)]


class RepairReq(ctypes.Structure):
    _fields_ = [("cache", ctypes.c_void_p), ("n_edits", ctypes.c_int32),
                ("edit_start", ctypes.c_void_p), ("edit_len", ctypes.c_void_p),
                ("new_tokens", ctypes.c_void_p), ("positions", ctypes.c_void_p),
                ("n_positions", ctypes.c_int32)]


_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_sigs = {
    "kvr_last_error": ([], ctypes.c_char_p),
    "kvr_set_allocator": ([_P, _P, _P], _I32),
    "kvr_model_create": ([ctypes.POINTER(ModelConfig), ctypes.POINTER(Weights), ctypes.c_uint64,
                          ctypes.POINTER(_P)], _I32),
    "kvr_model_free": ([_P], None),
    "kvr_model_set_stream": ([_P, _P], _I32),
    "kvr_synchronize": ([_P], _I32),
    "kvr_prefill": ([_P, _P, _I32, ctypes.POINTER(_P)], _I32),
    "kvr_cache_free": ([_P], None),
    "kvr_cache_load": ([_P, _P, _I32, _P, _P, ctypes.POINTER(_P)], _I32),
    "kvr_select": ([_P, _P, _I32, _I32, _I32, _I32, _P, ctypes.c_uint64, _P, _P], _I32),
    "kvr_repair": ([_P, _P, _I32, _I32, _P, _I32], _I32),
    "kvr_repair_read": ([_P, _P, _I32, _I32, _P, _I32, _P, _P], _I32),
    "kvr_repair_batch": ([_P, _P, _I32], _I32),
    "kvr_logits": ([_P, _P, _P, _I32, _P], _I32),
    "kvr_cache_len": ([_P], _I32),
    "kvr_cache_tokens": ([_P, _P], _I32),
    "kvr_cache_read": ([_P, _P, _I32, _I32, _I32, _P, _P], _I32),
    "kvr_cache_read_raw": ([_P, _P, _I32, _I32, _I32, _P, _P], _I32),
    "kvr_model_read_tensor": ([_P, ctypes.c_char_p, _I32, _P, ctypes.c_size_t], _I32),
    "kvr_profile_enable": ([_P, _I32], _I32),
    "kvr_profile_reset": ([_P], _I32),
    "kvr_profile_read": ([_P, _I32, _P, _P, _P, _P, _I32, _P], _I32),
    "kvr_launch_count": ([_P], ctypes.c_int64),
    "kvr_wait_probe": ([_P, _I32], _I32),
    "kvr_trace_enable": ([_P, _I32], _I32),
    "kvr_trace_read": ([_P, _P, _I32, _P], _I32),
    "kvr_linear": ([_P, ctypes.c_char_p, _I32, _P, _I32, _P], _I32),
    "kvr_linear_noalloc": ([_P, ctypes.c_char_p, _I32, _P, _I32, _P], _I32),
    "kvr_transplant": ([_P, _P, _P, _I32], _I32),
    "kvr_answer_logprob": ([_P, _P, _P, _I32, _P, _I32, _P], _I32),
    "kvr_margin": ([_P, _P, _P, _I32, _P, _I32, _P, _I32, _P], _I32),
}
for _name, (_args, _res) in _sigs.items():
    _f = getattr(_lib, _name)
    _f.argtypes = _args
    _f.restype = _res

EXPORTED = tuple(_sigs)


def _check(rc: int):
    if rc != KVR_OK:
        raise KvrError(rc, _lib.kvr_last_error().decode())


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _ptr(a: np.ndarray):
    return a.ctypes.data if a.size else None


def make_config(cfg: dict, max_context: int = 8192, max_rows: int = 4096) -> ModelConfig:
    return ModelConfig(cfg["vocab"], cfg["d_model"], cfg["n_layers"], cfg["n_heads"],
                       cfg["n_kv_heads"], cfg["head_dim"], cfg["ffn"],
                       1 if cfg.get("qkv_bias") else 0, DTYPES[cfg["dtype"]],
                       cfg.get("delim_id", 13), float(cfg["rope_theta"]), float(cfg["rms_eps"]),
                       int(max_context), int(max_rows))


class _WeightTables:
    def __init__(self, cfg: dict, W: dict):
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

        def table(key):
            arr = (ctypes.c_void_p * len(W["layers"]))(*[ptr(ly.get(key)) for ly in W["layers"]])
            self.keep.append(arr)
            return ctypes.cast(arr, _PP)

        self.s = Weights(ptr(W["embed"]), ptr(W["final_norm"]), ptr(W["lm_head"]),
                         table("attn_norm"), table("wq"), table("wk"), table("wv"), table("wo"),
                         table("bq"), table("bk"), table("bv"), table("mlp_norm"), table("wg"),
                         table("wu"), table("wd"))


# ------------------------------------------------ C entry points by name

def kvr_model_create(cfg: dict, weights: dict | None = None, seed: int = 0,
                     max_context: int = 8192, max_rows: int = 4096) -> ctypes.c_void_p:
    c = make_config(cfg, max_context, max_rows)
    out = ctypes.c_void_p()
    tabs = _WeightTables(cfg, weights) if weights is not None else None
    _check(_lib.kvr_model_create(ctypes.byref(c), ctypes.byref(tabs.s) if tabs else None,
                                 seed, ctypes.byref(out)))
    return out


def kvr_model_free(model):
    _lib.kvr_model_free(model)


def kvr_model_set_stream(model, stream_handle: int | None):
    _check(_lib.kvr_model_set_stream(model, stream_handle))


def kvr_synchronize(model):
    _check(_lib.kvr_synchronize(model))


def kvr_prefill(model, tokens) -> ctypes.c_void_p:
    t = _i32(tokens)
    out = ctypes.c_void_p()
    _check(_lib.kvr_prefill(model, _ptr(t), t.size, ctypes.byref(out)))
    return out


def kvr_cache_free(cache):
    _lib.kvr_cache_free(cache)


def kvr_cache_load(model, tokens, k, v, dtype) -> ctypes.c_void_p:
    """k, v: [n][n_layers][n_kv_heads][head_dim] in the cache's element type
    (uint16 bf16 bit patterns, or float32)."""
    t = _i32(tokens)
    k = np.ascontiguousarray(k)
    v = np.ascontiguousarray(v)
    for a in (k, v):
        if a.dtype != np.dtype(dtype) or a.shape[:1] != (t.size,):
            raise ValueError(f"cache rows must be {np.dtype(dtype)} [{t.size}, L, G, dh]")
    out = ctypes.c_void_p()
    _check(_lib.kvr_cache_load(model, _ptr(t), t.size, k.ctypes.data, v.ctypes.data,
                               ctypes.byref(out)))
    return out


def kvr_select(model, cache, policy: str, K: int, edit_start: int, new_tokens,
               seed: int = 0) -> np.ndarray:
    nt = _i32(new_tokens)
    out = np.zeros(max(K, 1), np.int32)
    cnt = ctypes.c_int32(0)
    _check(_lib.kvr_select(model, cache, POLICIES[policy], K, edit_start, nt.size, _ptr(nt),
                           seed & 0xFFFFFFFFFFFFFFFF, out.ctypes.data, ctypes.byref(cnt)))
    return out[:cnt.value].copy()


def kvr_repair(cache, new_tokens, edit_start: int, positions):
    nt, ps = _i32(new_tokens), _i32(positions)
    _check(_lib.kvr_repair(cache, _ptr(nt), edit_start, nt.size, _ptr(ps), ps.size))


def kvr_repair_read(cache, new_tokens, edit_start: int, positions, n_layers: int,
                    n_kv_heads: int, head_dim: int, dtype, k_out=None, v_out=None):
    """kvr_repair, returning the K and V rows of P (the span, then positions)
    as stored; k_out and v_out (optional, page-locked for the copies to
    overlap the pass) receive them in place."""
    nt, ps = _i32(new_tokens), _i32(positions)
    shape = (nt.size + ps.size, n_layers, n_kv_heads, head_dim)
    k = np.empty(shape, dtype) if k_out is None else k_out
    v = np.empty(shape, dtype) if v_out is None else v_out
    for a in (k, v):
        if a.shape != shape or a.dtype != np.dtype(dtype) or not a.flags.c_contiguous:
            raise ValueError(f"readback buffer must be C-contiguous {np.dtype(dtype)}{shape}")
    _check(_lib.kvr_repair_read(cache, _ptr(nt), edit_start, nt.size, _ptr(ps), ps.size,
                                k.ctypes.data, v.ctypes.data))
    return k, v


def kvr_repair_batch(model, reqs):
    """reqs: list of (cache, [(edit_start, new_tokens), ...], positions)."""
    keep, arr = [], (RepairReq * max(len(reqs), 1))()
    for i, (cache, edits, positions) in enumerate(reqs):
        st = _i32([e[0] for e in edits])
        ln = _i32([len(e[1]) for e in edits])
        nt = _i32(np.concatenate([np.asarray(e[1], np.int32) for e in edits])
                  if edits else np.zeros(0, np.int32))
        ps = _i32(positions)
        keep += [st, ln, nt, ps]
        arr[i] = RepairReq(cache, len(edits), _ptr(st), _ptr(ln), _ptr(nt), _ptr(ps), ps.size)
    _check(_lib.kvr_repair_batch(model, arr, len(reqs)))


def kvr_logits(model, cache, query, vocab: int) -> np.ndarray:
    q = _i32(query)
    out = np.zeros(vocab, np.float32)
    _check(_lib.kvr_logits(model, cache, _ptr(q), q.size, out.ctypes.data))
    return out


def kvr_transplant(dst, src, positions):
    ps = _i32(positions)
    _check(_lib.kvr_transplant(dst, src, _ptr(ps), ps.size))


def kvr_answer_logprob(model, cache, prompt, answer) -> float:
    pr, an = _i32(prompt), _i32(answer)
    out = ctypes.c_double(0.0)
    _check(_lib.kvr_answer_logprob(model, cache, _ptr(pr), pr.size, _ptr(an), an.size,
                                   ctypes.byref(out)))
    return out.value


def kvr_margin(model, cache, prompt, a_new, a_old) -> float:
    pr, an, ao = _i32(prompt), _i32(a_new), _i32(a_old)
    out = ctypes.c_double(0.0)
    _check(_lib.kvr_margin(model, cache, _ptr(pr), pr.size, _ptr(an), an.size, _ptr(ao),
                           ao.size, ctypes.byref(out)))
    return out.value


def kvr_cache_len(cache) -> int:
    return int(_lib.kvr_cache_len(cache))


def kvr_cache_tokens(cache) -> np.ndarray:
    out = np.zeros(kvr_cache_len(cache), np.int32)
    _check(_lib.kvr_cache_tokens(cache, out.ctypes.data))
    return out


def kvr_cache_read(cache, positions, layer_begin: int, layer_end: int, n_kv_heads: int,
                   head_dim: int):
    ps = _i32(positions)
    shape = (ps.size, layer_end - layer_begin, n_kv_heads, head_dim)
    k = np.zeros(shape, np.float32)
    v = np.zeros(shape, np.float32)
    _check(_lib.kvr_cache_read(cache, _ptr(ps), ps.size, layer_begin, layer_end,
                               k.ctypes.data, v.ctypes.data))
    return k, v


def kvr_cache_read_raw(cache, positions, layer_begin: int, layer_end: int, n_kv_heads: int,
                       head_dim: int, dtype, k_out=None, v_out=None):
    """K and V rows as stored (bf16 bit patterns as uint16, or float32); k_out and
    v_out (optional, e.g. page-locked) receive them in place."""
    ps = _i32(positions)
    shape = (ps.size, layer_end - layer_begin, n_kv_heads, head_dim)
    k = np.empty(shape, dtype) if k_out is None else k_out
    v = np.empty(shape, dtype) if v_out is None else v_out
    for a in (k, v):
        if a.shape != shape or a.dtype != np.dtype(dtype) or not a.flags.c_contiguous:
            raise ValueError(f"readback buffer must be C-contiguous {np.dtype(dtype)}{shape}")
    _check(_lib.kvr_cache_read_raw(cache, _ptr(ps), ps.size, layer_begin, layer_end,
                                   k.ctypes.data, v.ctypes.data))
    return k, v


def kvr_model_read_tensor(model, name: str, layer: int, shape, dtype) -> np.ndarray:
    out = np.zeros(shape, dtype)
    _check(_lib.kvr_model_read_tensor(model, name.encode(), layer, out.ctypes.data, out.nbytes))
    return out


def kvr_linear(model, name: str, layer: int, x: np.ndarray, n_out: int) -> np.ndarray:
    x = np.ascontiguousarray(x)
    y = np.zeros((x.shape[0], n_out), np.float32)
    _check(_lib.kvr_linear(model, name.encode(), layer, x.ctypes.data, x.shape[0],
                           y.ctypes.data))
    return y


def kvr_linear_noalloc(model, name: str, layer: int, x_dev_ptr: int, M: int, y_dev_ptr: int):
    """x_dev_ptr, y_dev_ptr: device addresses owned by the caller (e.g.
    torch tensors' data_ptr()); asynchronous on the model's stream."""
    _check(_lib.kvr_linear_noalloc(model, name.encode(), layer, x_dev_ptr, M, y_dev_ptr))


def kvr_profile_enable(model, enable: bool = True):
    _check(_lib.kvr_profile_enable(model, 1 if enable else 0))


def kvr_profile_reset(model):
    _check(_lib.kvr_profile_reset(model))


def kvr_profile_read(model) -> dict:
    cap = 64
    ms = np.zeros(cap, np.float64)
    la = np.zeros(cap, np.int64)
    by = np.zeros(cap, np.int64)
    names = ctypes.create_string_buffer(4096)
    n = ctypes.c_int32(0)
    _check(_lib.kvr_profile_read(model, cap, ms.ctypes.data, la.ctypes.data, by.ctypes.data,
                                 names, 4096, ctypes.byref(n)))
    labels = names.raw.split(b"\0")[:n.value]
    return {lab.decode(): dict(ms=float(ms[i]), launches=int(la[i]), bytes=int(by[i]))
            for i, lab in enumerate(labels)}


def kvr_trace_enable(model, capacity: int) -> None:
    _check(_lib.kvr_trace_enable(model, int(capacity)))


def kvr_trace_read(model, cap: int) -> np.ndarray:
    """Trace records as uint64 [n][16]: kind | smid << 8 | block << 16,
    start, wait return, end, marks 0..7, zeros (ns)."""
    out = np.zeros((max(cap, 1), 16), np.uint64)
    n = ctypes.c_int32(0)
    _check(_lib.kvr_trace_read(model, out.ctypes.data, int(cap), ctypes.byref(n)))
    return out[:min(n.value, cap)].copy()


def kvr_launch_count(model) -> int:
    return int(_lib.kvr_launch_count(model))


# ---------------------------------------------- torch caching allocator hook

_ALLOC = ctypes.CFUNCTYPE(ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p)
_FREE = ctypes.CFUNCTYPE(None, ctypes.c_void_p, ctypes.c_void_p)
_hooks = []
_live_models = weakref.WeakSet()


def _close_all():
    """Free every model still open (and with it its caches) while the
    allocator that gave them their device memory is still alive: at
    interpreter exit, finalisers otherwise run in no defined order."""
    for m in list(_live_models):
        m.close()


atexit.register(_close_all)


def use_torch_allocator():
    """Route the library's device allocations through PyTorch's caching
    allocator (call before creating a model)."""
    import torch

    def alloc(nbytes, ctx):
        try:
            return torch.cuda.caching_allocator_alloc(int(nbytes))
        except Exception:  # out of memory: the library reports KVR_E_NOMEM
            return None

    def free(ptr, ctx):
        if ptr:
            try:
                torch.cuda.caching_allocator_delete(ptr)
            except Exception:  # an exception cannot cross into the library
                pass

    a, f = _ALLOC(alloc), _FREE(free)
    _hooks[:] = [a, f]
    _check(_lib.kvr_set_allocator(ctypes.cast(a, _P), ctypes.cast(f, _P), None))
    # run before PyTorch's own exit handlers (registered at its import, earlier)
    atexit.unregister(_close_all)
    atexit.register(_close_all)


def use_cuda_allocator():
    _check(_lib.kvr_set_allocator(None, None, None))
    _hooks.clear()


# ------------------------------------------------------------ owners

class Model:
    def __init__(self, cfg: dict, weights: dict | None = None, seed: int = 0,
                 max_context: int = 8192, max_rows: int = 4096):
        self.cfg = dict(cfg)
        self._caches = weakref.WeakSet()
        self.h = kvr_model_create(cfg, weights, seed, max_context, max_rows)
        _live_models.add(self)

    def close(self):
        if getattr(self, "h", None):
            for c in list(self._caches):  # the library frees them with the model
                c.h = None
            kvr_model_free(self.h)
            self.h = None

    def __del__(self):
        self.close()

    def set_stream(self, stream_handle):
        kvr_model_set_stream(self.h, stream_handle)

    def synchronize(self):
        kvr_synchronize(self.h)

    def wait_probe(self, limit_us: int):
        """Enqueue a device wait that runs out after limit_us (see kvr_wait_probe)."""
        _check(_lib.kvr_wait_probe(self.h, int(limit_us)))

    def prefill(self, tokens) -> "Cache":
        return Cache(self, kvr_prefill(self.h, tokens))

    def load_cache(self, tokens, k, v) -> "Cache":
        """A cache holding the given K/V rows ([n][L][G][dh], cache dtype)."""
        dt = np.uint16 if self.cfg["dtype"] == "bf16" else np.float32
        return Cache(self, kvr_cache_load(self.h, tokens, k, v, dt))

    def select(self, cache: "Cache", policy: str, K: int, edit_start: int, new_tokens,
               seed: int = 0) -> np.ndarray:
        return kvr_select(self.h, cache.h, policy, K, edit_start, new_tokens, seed)

    def logits(self, cache: "Cache", query) -> np.ndarray:
        return kvr_logits(self.h, cache.h, query, self.cfg["vocab"])

    def answer_logprob(self, cache: "Cache", prompt, answer) -> float:
        return kvr_answer_logprob(self.h, cache.h, prompt, answer)

    def margin(self, cache: "Cache", prompt, a_new, a_old) -> float:
        """m_x of Eq. 2 for this cache state (kvr_margin)."""
        return kvr_margin(self.h, cache.h, prompt, a_new, a_old)

    def repair_batch(self, reqs):
        kvr_repair_batch(self.h, [(c.h, e, p) for c, e, p in reqs])

    def read_tensor(self, name: str, layer: int = 0) -> np.ndarray:
        c = self.cfg
        d, H, G, dh, F, V = (c["d_model"], c["n_heads"], c["n_kv_heads"], c["head_dim"],
                             c["ffn"], c["vocab"])
        shapes = dict(embed=(V, d), lm_head=(V, d), final_norm=(d,), wq=(H * dh, d),
                      wk=(G * dh, d), wv=(G * dh, d), wo=(d, H * dh), wg=(F, d), wu=(F, d),
                      wd=(d, F), bq=(H * dh,), bk=(G * dh,), bv=(G * dh,), attn_norm=(d,),
                      mlp_norm=(d,))
        dt = np.uint16 if c["dtype"] == "bf16" else np.float32
        return kvr_model_read_tensor(self.h, name, layer, shapes[name], dt)

    def trace_enable(self, capacity: int) -> None:
        """Attach a device timeline buffer of `capacity` records (0 detaches)."""
        self._trace_cap = int(capacity)
        kvr_trace_enable(self.h, capacity)

    def trace_read(self) -> np.ndarray:
        return kvr_trace_read(self.h, getattr(self, "_trace_cap", 0))

    def launches(self) -> int:
        return kvr_launch_count(self.h)


class Cache:
    def __init__(self, model: Model, handle):
        self.model = model
        self.h = handle
        model._caches.add(self)

    def close(self):
        if getattr(self, "h", None):
            # a freed model has freed its caches with it
            if getattr(self.model, "h", None):
                kvr_cache_free(self.h)
            self.h = None

    def __del__(self):
        self.close()

    @property
    def n(self) -> int:
        return kvr_cache_len(self.h)

    def repair(self, new_tokens, edit_start: int, positions):
        kvr_repair(self.h, new_tokens, edit_start, positions)

    def tokens(self) -> np.ndarray:
        return kvr_cache_tokens(self.h)

    def transplant_from(self, src: "Cache", positions):
        kvr_transplant(self.h, src.h, positions)

    def read(self, positions, layer_begin: int = 0, layer_end: int | None = None):
        c = self.model.cfg
        le = c["n_layers"] if layer_end is None else layer_end
        return kvr_cache_read(self.h, positions, layer_begin, le, c["n_kv_heads"], c["head_dim"])

    def repair_read(self, new_tokens, edit_start: int, positions, k_out=None, v_out=None):
        """repair, returning the K/V rows of P as stored (as read_raw over P)."""
        c = self.model.cfg
        dt = np.uint16 if c["dtype"] == "bf16" else np.float32
        return kvr_repair_read(self.h, new_tokens, edit_start, positions, c["n_layers"],
                               c["n_kv_heads"], c["head_dim"], dt, k_out, v_out)

    def read_raw(self, positions, layer_begin: int = 0, layer_end: int | None = None,
                 k_out=None, v_out=None):
        """Rows as stored: uint16 bf16 bit patterns for a bf16 model, else float32."""
        c = self.model.cfg
        le = c["n_layers"] if layer_end is None else layer_end
        dt = np.uint16 if c["dtype"] == "bf16" else np.float32
        return kvr_cache_read_raw(self.h, positions, layer_begin, le, c["n_kv_heads"],
                                  c["head_dim"], dt, k_out, v_out)
