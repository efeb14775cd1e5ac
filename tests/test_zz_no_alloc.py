"""kvr_linear_noalloc: a projection through the tensor-core GEMM that
allocates nothing during the call.

It exists for callers that must not allocate device memory while they run:
a serving loop under a memory budget reserved up front, code that cannot
take the device-wide synchronisation cudaMalloc/cudaFree may imply, or a
host whose allocator belongs to another framework.  Such a caller passes its
own device buffers; the GEMM's scratch sits in a fixed device array inside
the library.

The test checks it against kvr_linear, the entry point that runs the same
kernel with the same tiling and split but with scratch the library
allocated, so the results must be bit-identical: on two calls in a row, for
1, 40 and 64 rows.  wqkv, wo and wd (48 and 32 output tiles) take cluster
split-K, reduced in shared memory; lm_head (1002 output tiles, more than
the SMs) takes stream-K, whose split tiles go through the fixed array's
partials and counters.  It also checks that the calls allocate nothing (no
call into the library's allocator hook, free device memory unchanged), that
host pointers and sizes beyond the fixed scratch are refused.
"""
import ctypes

import numpy as np
import pytest

from paper_2609_17983_gb300 import synth

try:
    from paper_2609_17983_gb300 import kvrepair as kv
except ImportError as _e:  # pragma: no cover
    kv, _IMPORT_ERROR = None, _e

pytestmark = pytest.mark.gpu


def test_noalloc_matches_linear_and_allocates_nothing():
    if kv is None:
        raise _IMPORT_ERROR
    import torch
    calls = {"alloc": 0}

    # the library's allocations go through this hook (PyTorch's caching
    # allocator, counted) for the whole life of the model
    def alloc(nbytes, ctx):
        calls["alloc"] += 1
        try:
            return torch.cuda.caching_allocator_alloc(int(nbytes))
        except Exception:
            return None

    def free(ptr, ctx):
        if ptr:
            torch.cuda.caching_allocator_delete(ptr)

    hooks = (kv._ALLOC(alloc), kv._FREE(free))
    assert kv._lib.kvr_set_allocator(ctypes.cast(hooks[0], ctypes.c_void_p),
                                     ctypes.cast(hooks[1], ctypes.c_void_p), None) == 0
    model = None
    try:
        cfg = synth.preset("llama8b", n_layers=1)
        d, F, V = cfg["d_model"], cfg["ffn"], cfg["vocab"]
        model = kv.Model(cfg, None, seed=0, max_context=256, max_rows=64)
        shapes = [("wqkv", 6144, d), ("wo", d, d), ("wd", d, F), ("lm_head", V, d)]
        first = True
        for name, N, K in shapes:
            for M in (1, 40, 64):
                x = synth.tensor(1000 + M, 3, (M, K), "bf16", std=1.0)
                ref = kv.kvr_linear(model.h, name, 0, x, N)
                xd = torch.from_numpy(x.view(np.int16)).cuda()
                for call in range(2):
                    yd = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
                    torch.cuda.synchronize()
                    free0 = torch.cuda.mem_get_info()[0]
                    n0 = calls["alloc"]
                    kv.kvr_linear_noalloc(model.h, name, 0, xd.data_ptr(), M, yd.data_ptr())
                    model.synchronize()
                    assert calls["alloc"] == n0, (name, M, call)
                    # the first call may load the library's device code and
                    # array; every later one leaves free memory as it was
                    if not first:
                        assert torch.cuda.mem_get_info()[0] == free0, (name, M, call)
                    first = False
                    got = yd.cpu().numpy()
                    assert np.array_equal(got, ref), (name, M, call,
                                                      float(np.nanmax(np.abs(got - ref))))
        # sizes beyond the fixed scratch, and host memory, are refused
        xd = torch.zeros((65, d), dtype=torch.int16, device="cuda")
        yd = torch.zeros((65, d), dtype=torch.float32, device="cuda")
        with pytest.raises(kv.KvrError) as e:
            kv.kvr_linear_noalloc(model.h, "wo", 0, xd.data_ptr(), 65, yd.data_ptr())
        assert e.value.code == 6 and "64" in str(e.value)
        xh = np.zeros((8, d), np.uint16)
        yh = np.zeros((8, d), np.float32)
        with pytest.raises(kv.KvrError) as e:
            kv.kvr_linear_noalloc(model.h, "wo", 0, xh.ctypes.data, 8, yd.data_ptr())
        assert e.value.code == 1
        with pytest.raises(kv.KvrError) as e:
            kv.kvr_linear_noalloc(model.h, "wo", 0, xd.data_ptr(), 8, yh.ctypes.data)
        assert e.value.code == 1
        assert np.all(yh == 0)
    finally:
        if model is not None:
            model.close()  # freed through the hook it was allocated with
        kv.use_cuda_allocator()
