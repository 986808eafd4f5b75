"""rv_verify_head_static: the LM-head call for callers that cannot allocate
device memory (no handle, fixed internal scratch).  Its results must match
rv_verify_head's on the same inputs, on two calls in a row (the second call
must not see the first call's leftovers), within the tolerances of the parity
tests.  This file is collected last on purpose.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ALPHA = 0.3


@pytest.fixture(scope="module")
def env():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2505_18629_gb300 import build
    build.build()
    import tests.gpu_util as gu
    from paper_2505_18629_gb300 import rv, synth
    return gu, rv, synth


def _outputs(torch, B, g, rv):
    return (torch.full((B, g + 1, rv.RV_NSCORES), float("nan"), device="cuda"),
            torch.full((B, g + 1), -7, dtype=torch.int32, device="cuda"),
            torch.full((B, g), float("nan"), device="cuda"))


def _inputs(gu, synth, seed, B, gamma, R, V, H):
    wl = synth.Workload("static", B=B, gamma=gamma, R=R, ctx=(4, 4), H=H, Hq=4, Hkv=4, D=64,
                        V=V, dtype="bf16", p_argmax=0.7, seed=seed)
    inp = synth.generate(wl, with_cache=False)
    drafts = gu.oracle_drafts(inp, ALPHA)
    return wl, inp, drafts


def test_static_head_matches_handle_head_on_two_calls(env):
    import torch
    gu, rv, synth = env
    cases = [_inputs(gu, synth, 61, B=3, gamma=5, R=6, V=1500, H=512),
             _inputs(gu, synth, 62, B=2, gamma=4, R=3, V=1500, H=512)]
    W = gu.to_dev(cases[0][1].W)                         # same weight, different rows/drafts
    h = rv.rv_create(512, 1500, 4, 4, 64, 3, 5, 6, 64, rv.RV_DTYPE_BF16)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for wl, inp, drafts in cases:
        hid, d = gu.to_dev(inp.hidden), gu.to_dev(drafts.astype(np.int32))
        ref = _outputs(torch, wl.B, wl.gamma, rv)
        rv.rv_verify_head(h, hid, W, d, wl.gamma, wl.R, ALPHA, *ref)
        got = _outputs(torch, wl.B, wl.gamma, rv)
        rv.rv_verify_head_static(hid, W, d, wl.gamma, wl.R, ALPHA, *got, dev_status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        sr, sg = gu.to_np(ref[0]), gu.to_np(got[0])
        np.testing.assert_allclose(sg[..., :3], sr[..., :3], atol=gu.LOGP_ATOL, rtol=0)
        np.testing.assert_allclose(sg[:, :-1, 3:], sr[:, :-1, 3:], atol=gu.LOGP_ATOL, rtol=0)
        assert np.isnan(sg[:, -1, 3:6]).all()                 # no draft at the bonus position
        np.testing.assert_allclose(sg[..., 6], sr[..., 6], atol=gu.LOGP_ATOL, rtol=0)  # entropy
        np.testing.assert_allclose(gu.to_np(got[2]), gu.to_np(ref[2]), atol=gu.LOGP_ATOL, rtol=0)
        close = gu.to_np(ref[2]) < gu.MARGIN_EPS
        am_r, am_g = gu.to_np(ref[1]), gu.to_np(got[1])
        assert ((am_r == am_g)[:, :-1] | close).all() and (am_r[:, -1] == am_g[:, -1]).all()
    h.close()


def test_static_head_rejects_sizes_beyond_its_scratch(env):
    import torch
    gu, rv, synth = env
    z = torch.zeros(16, device="cuda")
    zi = torch.zeros(16, dtype=torch.int32, device="cuda")
    big_b = torch.zeros((rv.RV_STATIC_MAX_PAIRS // 4 + 1, 12, 64), dtype=torch.bfloat16,
                        device="cuda")
    w = torch.zeros((256, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(rv.RVError) as e:           # B * (gamma + 1) = 17 * 4 > 64 pairs
        rv.rv_verify_head_static(big_b, w, zi, 3, 5, ALPHA, z, zi, z)
    assert e.value.code == rv.RV_ERR_CAPACITY
    wide = torch.zeros((256, rv.RV_STATIC_MAX_HIDDEN + 8), dtype=torch.bfloat16, device="cuda")
    hid = torch.zeros((1, 12, rv.RV_STATIC_MAX_HIDDEN + 8), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(rv.RVError) as e:
        rv.rv_verify_head_static(hid, wide, zi, 3, 5, ALPHA, z, zi, z)
    assert e.value.code == rv.RV_ERR_CAPACITY
