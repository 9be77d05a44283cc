"""The C-ABI library loads, exports every symbol include/ssd.h declares, and
rejects bad arguments on the host before touching a GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "ssd.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ssd_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def ssd():
    import __graft_entry__ as g
    g._lib_builder().build()
    import paper_2309_08168_gb300 as m
    return m


def test_exports_every_declared_symbol(ssd):
    names = _declared()
    assert len(names) == 14
    assert sorted(ssd.EXPORTS) == names
    lib = ctypes.CDLL(ssd.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n


def test_struct_layouts_match_header(ssd):
    # ssd_config: 8 ints + 2 floats; ssd_stats: 4 ints, double, 33 ints, 3 floats, long long, float
    assert ctypes.sizeof(ssd.ssd_config) == 40
    assert ctypes.sizeof(ssd.ssd_weights) == 8 * 12 + 8
    assert ssd.ssd_stats.accept_rate.offset == 16
    assert ssd.ssd_stats.hist.offset == 24
    assert ssd.ssd_stats.total_ms.offset == 24 + 33 * 4 + 8
    assert ssd.ssd_stats.kernel_launches.offset == 168
    assert ssd.ssd_stats.gamma.offset == 176 and ctypes.sizeof(ssd.ssd_stats) == 184


def _cfg(ssd, **kw):
    base = dict(n_layers=2, d_model=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688, vocab=2048, max_seq=64)
    base.update(kw)
    return ssd.make_config(**base)


@pytest.mark.parametrize("bad", [dict(head_dim=96), dict(n_kv_heads=3), dict(d_model=200), dict(d_model=320),
                                 dict(ffn=100), dict(vocab=40000), dict(max_seq=1), dict(n_layers=0),
                                 dict(n_heads=3, n_kv_heads=1)])
def test_create_rejects_bad_config(ssd, bad):
    w = ssd.ssd_weights()  # all NULL: config is checked first, no device touched
    with pytest.raises(ssd.SSDError) as e:
        ssd.ssd_create(_cfg(ssd, **bad), w)
    assert e.value.code == ssd.SSD_ERR_INVALID_ARG
    assert ssd.ssd_last_error()


def test_create_rejects_null_weights(ssd):
    with pytest.raises(ssd.SSDError) as e:
        ssd.ssd_create(_cfg(ssd), ssd.ssd_weights())
    assert e.value.code == ssd.SSD_ERR_INVALID_ARG
    assert "NULL" in str(e.value)


def test_noalloc_rejects_bad_sizes_on_host(ssd):
    lib = ssd.lib
    # NULL pointers and sizes are rejected before any device work
    assert lib.ssd_linear_noalloc(None, None, None, 64, 64, 1, None) == ssd.SSD_ERR_INVALID_ARG
    buf = (ctypes.c_float * 64)()
    p = ctypes.addressof(buf) & ~15
    assert lib.ssd_linear_noalloc(p, p, p, 64, 40, 1, None) == ssd.SSD_ERR_INVALID_ARG  # K % 16
    assert lib.ssd_linear_noalloc(p, p, p, 64, 64, 17, None) == ssd.SSD_ERR_INVALID_ARG  # M > 16
    assert lib.ssd_linear_noalloc(p, p, p, 4097 * 64, 64, 1, None) == ssd.SSD_ERR_CAPACITY  # tiles
    assert lib.ssd_linear_noalloc(p, p, p, 32000, 8192, 16, None) == ssd.SSD_ERR_CAPACITY  # scratch
    assert "scratch" in ssd.ssd_last_error()


def test_null_handle_calls_fail_cleanly(ssd):
    lib = ssd.lib
    assert lib.ssd_set_skip(None, None, 0) == ssd.SSD_ERR_INVALID_ARG
    assert lib.ssd_set_sampling(None, 1.0, 1.0) == ssd.SSD_ERR_INVALID_ARG
    assert lib.ssd_set_draft_exit(None, 1, 0.6, 0.9, 0.01, 0.5, 0.9) == ssd.SSD_ERR_INVALID_ARG
    assert lib.ssd_prefill(None, None, 1) == ssd.SSD_ERR_INVALID_ARG
    assert lib.ssd_generate(None, None, 0, 1, 0, 0, 0, None, None) == ssd.SSD_ERR_INVALID_ARG
    lib.ssd_destroy(None)
