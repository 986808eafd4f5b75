"""The binding refuses mis-shaped or mis-typed tensors before it calls the C
library (which sees only pointers and could read past a short buffer on the
device).  CPU only: the checks run before any handle pointer is used, so a
handle object that owns no library handle is enough."""
import pytest
import torch


@pytest.fixture(scope="module")
def rv():
    from paper_2505_18629_gb300 import build
    build.build()
    from paper_2505_18629_gb300 import rv as rvmod
    return rvmod


def _handle(rv, dtype=None):
    cfg = rv.rv_config(320, 1000, 8, 2, 128, 3, 4, 5, 400,
                       rv.RV_DTYPE_BF16 if dtype is None else dtype)
    return rv.Handle(None, cfg)          # owns nothing; .ptr would raise


def _head_args(rv, B=2, g=4, R=5, rows=None, H=320, V=1000, dt=torch.bfloat16):
    rows = 2 * g + R + 1 if rows is None else rows
    return (torch.zeros((B, rows, H), dtype=dt), torch.zeros((V, H), dtype=dt),
            torch.zeros((B, g), dtype=torch.int32), g, R, 0.3,
            torch.zeros((B, g + 1, rv.RV_NSCORES)), torch.zeros((B, g + 1), dtype=torch.int32),
            torch.zeros((B, g)))


def test_head_refuses_short_hidden(rv):
    h = _handle(rv)
    with pytest.raises(ValueError, match="hidden has shape"):
        rv.rv_verify_head(h, *_head_args(rv, rows=13))


def test_head_refuses_wrong_width_weight_and_dtype(rv):
    h = _handle(rv)
    args = list(_head_args(rv))
    args[1] = torch.zeros((1000, 256), dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="w_head has shape"):
        rv.rv_verify_head(h, *args)
    with pytest.raises(ValueError, match="dtype"):
        rv.rv_verify_head(h, *_head_args(rv, dt=torch.float32))


def test_head_refuses_host_tensors_where_device_memory_is_expected(rv):
    h = _handle(rv)
    with pytest.raises(ValueError, match="device memory"):
        rv.rv_verify_head(h, *_head_args(rv))     # right shapes, but host tensors


def test_head_output_shapes_are_checked(rv):
    h = _handle(rv)
    args = list(_head_args(rv))
    args[6] = torch.zeros((2, 5, 3))              # scores with too few fields
    with pytest.raises(ValueError, match="scores"):
        rv.rv_verify_head(h, *args)


def test_standard_mode_takes_gamma_plus_one_rows(rv):
    h = _handle(rv)
    h.head_mode = rv.RV_HEAD_STANDARD
    # the reflective layout's rows are refused in standard mode (gamma + 1 rows expected)
    with pytest.raises(ValueError, match=r"hidden has shape \[2, 14, 320\], expected \[2, 5, 320\]"):
        rv.rv_verify_head(h, *_head_args(rv))


def test_static_head_refuses_short_hidden(rv):
    hid, w, d, g, R, a, sc, am, mg = _head_args(rv, rows=12)
    with pytest.raises(ValueError, match="hidden has shape"):
        rv.rv_verify_head_static(hid, w, d, g, R, a, sc, am, mg)
    hid, w, d, g, R, a, sc, am, mg = _head_args(rv)
    with pytest.raises(ValueError, match="draft_ids"):
        rv.rv_verify_head_static(hid, w, torch.zeros((2, 3), dtype=torch.int32), g, R, a, sc,
                                 am, mg)


def test_step_checks_cache_and_block_shapes(rv):
    h = _handle(rv)
    B, g, R = 2, 4, 5
    Lb = 2 * g + R
    bf = torch.bfloat16
    i32 = torch.int32
    q = torch.zeros((B, Lb, 8, 128), dtype=bf)
    kb = torch.zeros((B, Lb, 2, 128), dtype=bf)
    kc = torch.zeros((B, 2, 399, 128), dtype=bf)  # capacity one short of max_ctx = 400
    hid, w, d, _, _, _, sc, am, mg = _head_args(rv)
    prompt = torch.zeros((1,), dtype=i32)
    prefix = torch.zeros((B, 4), dtype=i32)
    ctx = torch.zeros((B,), dtype=i32)
    outs = (torch.zeros((B, Lb), dtype=i32), torch.zeros((B, Lb), dtype=i32), torch.zeros_like(q),
            sc, am, mg, torch.zeros((B, g), dtype=torch.uint8), torch.zeros((B,), dtype=i32),
            torch.zeros((B,), dtype=i32), torch.zeros((B,), dtype=i32))
    with pytest.raises(ValueError, match="k_cache"):
        rv.rv_verify_step(h, q, kb, kb, kc, kc, hid, w, d, prompt, prefix, ctx, 0.3, *outs)
