"""rv_verify_head_static: the LM-head call for callers that cannot allocate
device memory (no handle, fixed internal scratch).

Its results must match the oracle's verify_head and rv_verify_head's on the
same inputs, within the tolerances of the parity tests, on two calls in a row
(the second call must not see the first call's leftovers in the shared
scratch), with and without a caller-supplied status word, and at the 8B shape
(H = 4096, V = 128256, B = 1, gamma = 5, template 8), and at its limits
(64 pairs, H = 8192) without allocating.  This file is collected last on purpose.
"""
import numpy as np
import pytest

import oracle.rv_oracle as orc

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


def _check_against_oracle_and_handle(gu, rv, wl, inp, drafts, got, ref):
    """`got`: rv_verify_head_static's outputs; `ref`: rv_verify_head's."""
    sg, am_g, mg_g = (gu.to_np(t) for t in got)
    head = orc.verify_head(inp.W, inp.hidden, drafts, wl.gamma, wl.R, ALPHA)
    gu.compare_head(head, sg, am_g, mg_g, wl.gamma)
    # and the existing entry point on the same inputs
    sr, am_r, mg_r = (gu.to_np(t) for t in ref)
    np.testing.assert_allclose(sg[..., :3], sr[..., :3], atol=gu.LOGP_ATOL, rtol=0)
    np.testing.assert_allclose(sg[:, :-1, 3:], sr[:, :-1, 3:], atol=gu.LOGP_ATOL, rtol=0)
    np.testing.assert_allclose(sg[..., 6], sr[..., 6], atol=gu.LOGP_ATOL, rtol=0)  # entropy
    np.testing.assert_allclose(mg_g, mg_r, atol=gu.LOGP_ATOL, rtol=0)
    close = head["choice_gap"] < gu.MARGIN_EPS
    assert ((am_r == am_g) | close).all()


def test_static_head_matches_oracle_and_handle_head_on_two_calls(env):
    import torch
    gu, rv, synth = env
    cases = [_inputs(gu, synth, 61, B=3, gamma=5, R=6, V=1500, H=512),
             _inputs(gu, synth, 62, B=2, gamma=4, R=3, V=1500, H=512)]
    W = gu.to_dev(cases[0][1].W)                         # same weight, different rows/drafts
    h = rv.rv_create(512, 1500, 4, 4, 64, 3, 5, 6, 64, rv.RV_DTYPE_BF16)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for use_status in (True, False):
        for wl, inp, drafts in cases:
            inp.W = cases[0][1].W
            hid, d = gu.to_dev(inp.hidden), gu.to_dev(drafts.astype(np.int32))
            ref = _outputs(torch, wl.B, wl.gamma, rv)
            rv.rv_verify_head(h, hid, W, d, wl.gamma, wl.R, ALPHA, *ref)
            got = _outputs(torch, wl.B, wl.gamma, rv)
            rv.rv_verify_head_static(hid, W, d, wl.gamma, wl.R, ALPHA, *got,
                                     dev_status=status if use_status else None)
            torch.cuda.synchronize()
            assert int(status.item()) == 0
            _check_against_oracle_and_handle(gu, rv, wl, inp, drafts, got, ref)
    h.close()


def test_static_head_reports_draft_range_to_the_callers_status(env):
    import torch
    gu, rv, synth = env
    wl, inp, drafts = _inputs(gu, synth, 63, B=2, gamma=3, R=4, V=1500, H=512)
    bad = drafts.copy()
    bad[1, 2] = wl.V + 5                                  # out of range
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    got = _outputs(torch, wl.B, wl.gamma, rv)
    rv.rv_verify_head_static(gu.to_dev(inp.hidden), gu.to_dev(inp.W),
                             gu.to_dev(bad.astype(np.int32)), wl.gamma, wl.R, ALPHA, *got,
                             dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) & rv.RV_DEV_DRAFT_RANGE
    # the in-range positions are still scored as the oracle scores them
    sg = gu.to_np(got[0])
    head = orc.verify_head(inp.W, inp.hidden, drafts, wl.gamma, wl.R, ALPHA)
    np.testing.assert_allclose(sg[..., :3], np.stack([head["lse_orig"], head["lse_refl"],
                                                      head["lse_fused"]], -1),
                               atol=gu.LOGP_ATOL, rtol=0)
    np.testing.assert_allclose(sg[0, :wl.gamma, 3], head["logp_fused"][0], atol=gu.LOGP_ATOL)


def test_static_head_at_the_8b_shape(env):
    import torch
    gu, rv, synth = env
    wl = synth.WORKLOADS["llama3-8b-b1"]
    inp = synth.generate(wl, with_cache=False)
    drafts = gu.oracle_drafts(inp, ALPHA)
    W, hid = gu.to_dev(inp.W), gu.to_dev(inp.hidden)
    d = gu.to_dev(drafts.astype(np.int32))
    h = gu.make_handle(wl)
    ref = _outputs(torch, wl.B, wl.gamma, rv)
    rv.rv_verify_head(h, hid, W, d, wl.gamma, wl.R, ALPHA, *ref)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for _ in range(2):
        got = _outputs(torch, wl.B, wl.gamma, rv)
        rv.rv_verify_head_static(hid, W, d, wl.gamma, wl.R, ALPHA, *got, dev_status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        _check_against_oracle_and_handle(gu, rv, wl, inp, drafts, got, ref)
    h.close()


def test_static_head_at_its_limits_allocates_nothing(env):
    """64 pairs (B = 8, gamma = 7) at H = RV_STATIC_MAX_HIDDEN: the largest call
    it accepts.  After a first call (which may load the library's module), two
    more calls leave the device's free memory and the caching allocator's
    allocation count unchanged."""
    import torch
    gu, rv, synth = env
    B, gamma = 8, rv.RV_STATIC_MAX_PAIRS // 8 - 1
    wl, inp, drafts = _inputs(gu, synth, 64, B=B, gamma=gamma, R=4, V=1200,
                              H=rv.RV_STATIC_MAX_HIDDEN)
    assert B * (gamma + 1) == rv.RV_STATIC_MAX_PAIRS
    hid, W = gu.to_dev(inp.hidden), gu.to_dev(inp.W)
    d = gu.to_dev(drafts.astype(np.int32))
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    outs = [_outputs(torch, B, gamma, rv) for _ in range(3)]
    rv.rv_verify_head_static(hid, W, d, gamma, wl.R, ALPHA, *outs[0], dev_status=status)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    n0 = torch.cuda.memory_stats().get("allocation.all.allocated", 0)
    for got in outs[1:]:
        rv.rv_verify_head_static(hid, W, d, gamma, wl.R, ALPHA, *got, dev_status=status)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert torch.cuda.memory_stats().get("allocation.all.allocated", 0) == n0
    assert int(status.item()) == 0
    head = orc.verify_head(inp.W, inp.hidden, drafts, wl.gamma, wl.R, ALPHA)
    for got in outs:
        sg, am_g, mg_g = (gu.to_np(t) for t in got)
        gu.compare_head(head, sg, am_g, mg_g, wl.gamma)


def test_static_head_rejects_sizes_beyond_its_scratch(env):
    import torch
    gu, rv, synth = env
    bf, i32 = torch.bfloat16, torch.int32

    def call(B, gamma, R, V, H):
        hid = torch.zeros((B, 2 * gamma + R + 1, H), dtype=bf, device="cuda")
        w = torch.zeros((V, H), dtype=bf, device="cuda")
        d = torch.zeros((B, gamma), dtype=i32, device="cuda")
        rv.rv_verify_head_static(hid, w, d, gamma, R, ALPHA, *_outputs(torch, B, gamma, rv))

    with pytest.raises(rv.RVError) as e:           # B * (gamma + 1) = 17 * 4 > 64 pairs
        call(rv.RV_STATIC_MAX_PAIRS // 4 + 1, 3, 5, 256, 64)
    assert e.value.code == rv.RV_ERR_CAPACITY
    with pytest.raises(rv.RVError) as e:           # hidden size above the scratch rows
        call(1, 3, 5, 256, rv.RV_STATIC_MAX_HIDDEN + 8)
    assert e.value.code == rv.RV_ERR_CAPACITY
