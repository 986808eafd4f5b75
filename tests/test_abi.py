"""The C-ABI library loads, exports every entry point of include/rv.h, and
rejects bad arguments on the host before touching a GPU (no compute here)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "rv.h")


@pytest.fixture(scope="module")
def rv():
    from paper_2505_18629_gb300 import build
    build.build()
    from paper_2505_18629_gb300 import rv as rvmod
    return rvmod


def _declared():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"RV_API\s+[\w\s\*]+?\b(rv_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("rv_create", "rv_destroy", "rv_verify_attention", "rv_verify_head", "rv_accept",
              "rv_pack_block", "rv_verify_step", "rv_verify_step_host", "rv_read_status"):
        assert n in names


def test_library_exports_every_declared_symbol(rv):
    lib = ctypes.CDLL(rv.LIB_PATH)
    for n in _declared():
        assert hasattr(lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", rv.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT\s+(rv_\w+)", out))
    assert set(_declared()) <= exported
    # nothing but the C ABI is exported under the rv_ prefix
    assert exported <= set(_declared())


def test_binding_names_match_the_abi(rv):
    for n in _declared():
        if n in ("rv_last_error", "rv_destroy"):
            continue
        assert callable(getattr(rv, n)), n


def _cfg(rv, **kw):
    base = dict(hidden=256, vocab=4096, n_q_heads=4, n_kv_heads=4, head_dim=64, max_batch=2,
                max_gamma=4, max_template=4, max_ctx=128, dtype=rv.RV_DTYPE_F32)
    base.update(kw)
    return rv.rv_config(*[base[f] for f, _ in rv.rv_config._fields_])


@pytest.mark.parametrize("bad,code", [
    (dict(dtype=7), -1),
    (dict(hidden=0), -1),
    (dict(hidden=100), -2),                 # not a multiple of 8
    (dict(n_q_heads=6, n_kv_heads=4), -2),  # GQA groups must divide
    (dict(dtype=0, head_dim=96), -5),       # bf16 attention built for 64 / 128
    (dict(max_gamma=65), -3),
])
def test_create_rejects_bad_config_on_host(rv, bad, code):
    cfg = _cfg(rv, **bad)
    out = ctypes.c_void_p()
    rc = rv.lib().rv_create(ctypes.byref(cfg), ctypes.byref(out))
    assert rc == code
    assert out.value is None
    assert rv.lib().rv_last_error(None).decode() != ""


def test_create_null_arguments(rv):
    out = ctypes.c_void_p()
    assert rv.lib().rv_create(None, ctypes.byref(out)) == rv.RV_ERR_INVALID_ARG
    cfg = _cfg(rv)
    assert rv.lib().rv_create(ctypes.byref(cfg), None) == rv.RV_ERR_INVALID_ARG


def test_entry_points_reject_null_handle(rv):
    L = rv.lib()
    assert L.rv_verify_head(None, None, None, None, 1, 1, 0, 0.3, None, None, None, None) == -1
    assert L.rv_verify_attention(None, None, None, None, None, None, None, 1, 1, None, None) == -1
    assert L.rv_accept(None, None, None, 1, 1, None, None, None, None, None, None) == -1
    assert L.rv_pack_block(None, None, None, None, None, 1, 1, 0, 0, None, None, None) == -1
    assert L.rv_accept_typical(None, None, None, None, 1, 1, 0.09, 0.3, None, None, None, None,
                               None, None) == -1
    assert L.rv_set_acceptance(None, 1, 0.09, 0.3) == -1
    assert L.rv_accept_speculative(None, None, None, None, None, None, 1, 1, None, None, None,
                                   None, None, None) == -1
    assert L.rv_set_head_mode(None, 1) == -1
    assert L.rv_host_step_graphed(None, None) == -1
    assert L.rv_accept_sampled(None, None, None, 1.0, 1, 1, None, None, None, None, None,
                               None, None) == -1
    assert L.rv_pack_block_pending(None, None, None, None, None, None, 1, 1, 0, 0, None, None,
                                   None) == -1
    assert L.rv_destroy(None) == 0


@pytest.mark.skipif(__import__("torch").cuda.is_available(), reason="checks the no-GPU path")
def test_create_without_gpu_fails_cleanly(rv):
    cfg = _cfg(rv)
    out = ctypes.c_void_p()
    rc = rv.lib().rv_create(ctypes.byref(cfg), ctypes.byref(out))
    assert rc in (rv.RV_ERR_CUDA, rv.RV_ERR_UNSUPPORTED)
    assert out.value is None


def test_binding_constants_match_the_header():
    # every integer constant of include/rv.h has the same value in the binding
    from paper_2505_18629_gb300 import rv as rvmod
    text = open(HEADER).read()
    consts = {}
    for name, val in re.findall(r"^#define\s+(RV_\w+)\s+(\(?-?\d+\)?u?)\b", text, flags=re.M):
        consts[name] = int(val.strip("()u"))
    assert "RV_ACCEPT_TYPICAL_SAMPLED" in consts and "RV_SCORE_ENT_ORIG" in consts
    missing = [n for n in consts if not hasattr(rvmod, n)]
    assert not missing, missing
    wrong = {n: (getattr(rvmod, n), v) for n, v in consts.items() if getattr(rvmod, n) != v}
    assert not wrong, wrong
