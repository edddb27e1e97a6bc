"""The C-ABI library builds, loads and exports every symbol of include/*.h.

No compute call runs here (no GPU); only host-side argument validation,
which returns before any CUDA call, is exercised.
"""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__ as g
    g.build()
    from paper_2606_10820_gb300 import kforcing as kf
    return kf.load_library()


def declared_symbols():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^\s*(?:const\s+)?\w+\s*\*?\s*(kf_\w+)\s*\(", src, re.M):
            names.add(m.group(1))
    return sorted(names)


def test_header_declares_the_boundary():
    names = declared_symbols()
    for n in ("kf_init", "kf_prefill", "kf_decode_step", "kf_debug_logits", "kf_free",
              "kf_last_error"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in declared_symbols() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_uses_the_c_names(lib):
    from paper_2606_10820_gb300 import kforcing as kf
    for n in declared_symbols():
        if n.startswith("kf_op_"):
            continue
        assert hasattr(kf, n), n


def test_struct_layout_matches_header():
    from paper_2606_10820_gb300 import kforcing as kf
    # 16 int32 fields, 4 floats, then mtp_k; 15 pointers
    assert ctypes.sizeof(kf.kf_config) == 21 * 4
    assert ctypes.sizeof(kf.kf_weights) == 15 * ctypes.sizeof(ctypes.c_void_p)


def test_init_rejects_bad_config_on_host(lib):
    from paper_2606_10820_gb300 import kforcing as kf
    from synth import TINY
    cfg = kf.make_config(TINY, max_batch=2, max_k=2)
    cfg.d_model = 100          # not 64 * n_head
    with pytest.raises(kf.KfError) as e:
        kf.kf_init(cfg, {})
    assert e.value.code == kf.KF_E_ARG
    cfg = kf.make_config(TINY, max_batch=2, max_k=9)
    with pytest.raises(kf.KfError) as e:
        kf.kf_init(cfg, {})
    assert e.value.code == kf.KF_E_ARG
    assert "max_k" in kf.kf_last_error() or "NULL" in kf.kf_last_error()


def test_calls_on_null_context_fail_cleanly(lib):
    from paper_2606_10820_gb300 import kforcing as kf
    assert lib.kf_decode_step(None, 1, 1, None, None) == kf.KF_E_ARG
    assert lib.kf_prefill(None, 1, None, None) == kf.KF_E_ARG
    assert lib.kf_free(None) == kf.KF_OK
