"""kvr_linear_noalloc: a projection through the tensor-core GEMM that
allocates nothing during the call.

It exists for callers that must not allocate device memory while they run:
a serving loop under a memory budget reserved up front, code that cannot
take the device-wide synchronisation cudaMalloc/cudaFree may imply, or a
host whose allocator belongs to another framework.  Such a caller passes its
own device buffers; the GEMM's scratch sits in a fixed device array inside
the library.  The test checks it against kvr_linear, the entry point that
runs the same kernel with scratch the library allocated, on two calls in a
row, and checks that sizes beyond the fixed scratch are refused.
"""
import numpy as np
import pytest

from paper_2609_17983_gb300 import synth

try:
    from paper_2609_17983_gb300 import kvrepair as kv
except ImportError as _e:  # pragma: no cover
    kv, _IMPORT_ERROR = None, _e

pytestmark = pytest.mark.gpu


def rel(a, b):
    return float(np.abs(a - b).max() / np.abs(b).max())


def test_noalloc_matches_linear_on_two_calls_in_a_row():
    if kv is None:
        raise _IMPORT_ERROR
    import torch
    cfg = synth.preset("llama8b", n_layers=1)
    d, F, V = cfg["d_model"], cfg["ffn"], cfg["vocab"]
    model = kv.Model(cfg, None, seed=0, max_context=256, max_rows=64)
    shapes = [("wqkv", 6144, d), ("wo", d, d), ("wd", d, F), ("lm_head", V, d)]
    for name, N, K in shapes:
        for call, M in enumerate((40, 64)):
            x = synth.tensor(1000 + call, 3, (M, K), "bf16", std=1.0)
            ref = kv.kvr_linear(model.h, name, 0, x, N)
            xd = torch.from_numpy(x.view(np.int16)).cuda()
            yd = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
            torch.cuda.synchronize()
            kv.kvr_linear_noalloc(model.h, name, 0, xd.data_ptr(), M, yd.data_ptr())
            model.synchronize()
            got = yd.cpu().numpy()
            assert np.isfinite(got).all(), (name, call)
            assert rel(got, ref) <= 1e-3, (name, call)
    xd = torch.zeros((65, d), dtype=torch.int16, device="cuda")
    yd = torch.zeros((65, d), dtype=torch.float32, device="cuda")
    with pytest.raises(kv.KvrError) as e:
        kv.kvr_linear_noalloc(model.h, "wo", 0, xd.data_ptr(), 65, yd.data_ptr())
    assert e.value.code == 6 and "64" in str(e.value)
    model.close()
