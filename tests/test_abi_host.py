"""Host-side checks of the C ABI: the library loads, exports every entry point
that include/kvrepair.h declares, and rejects bad arguments before any device
work (no GPU needed)."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "kvrepair.h")


@pytest.fixture(scope="module")
def kv():
    from paper_2609_17983_gb300 import build
    build.build()
    from paper_2609_17983_gb300 import kvrepair
    return kvrepair


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = set(re.findall(r"\b(kvr_[a-z_]+)\s*\(", src))
    return sorted(n for n in names if not n.endswith("_fn"))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("kvr_model_create", "kvr_prefill", "kvr_select", "kvr_repair", "kvr_logits",
              "kvr_repair_batch", "kvr_cache_free", "kvr_model_free", "kvr_last_error"):
        assert n in names


def test_library_exports_every_declared_symbol(kv):
    lib = ctypes.CDLL(kv.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing
    assert set(declared_functions()) <= set(kv.EXPORTED) | {"kvr_last_error"}


def test_invalid_config_rejected_on_host(kv):
    from paper_2609_17983_gb300 import synth
    bad = synth.preset("tiny", n_kv_heads=3)
    with pytest.raises(kv.KvrError) as e:
        kv.kvr_model_create(bad)
    assert e.value.code == 1 and "multiple" in str(e.value)
    with pytest.raises(kv.KvrError) as e:
        kv.kvr_model_create(synth.preset("tiny", head_dim=96))
    assert e.value.code == 6


def test_null_handles_rejected(kv):
    lib = kv._lib
    assert lib.kvr_repair(None, None, 0, 0, None, 0) == 1
    assert lib.kvr_repair_read(None, None, 0, 0, None, 0, None, None) == 1
    one = np.array([5], np.int32)
    assert lib.kvr_repair_read(None, None, 0, 0, one.ctypes.data, 1, None, None) == 1
    assert b"k_out" in lib.kvr_last_error()
    assert lib.kvr_prefill(None, None, 0, None) == 1
    assert lib.kvr_select(None, None, 0, 1, 0, 0, None, 0, None, None) == 1
    assert lib.kvr_logits(None, None, None, 1, None) == 1
    assert lib.kvr_wait_probe(None, 1000) == 1
    assert lib.kvr_cache_load(None, None, 0, None, None, None) == 1
    assert lib.kvr_margin(None, None, None, 1, None, 1, None, 1, None) == 1
    assert lib.kvr_synchronize(None) == 1
    assert b"NULL" in lib.kvr_last_error()
    assert lib.kvr_cache_len(None) == -1
