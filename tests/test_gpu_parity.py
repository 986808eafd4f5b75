"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle.

Small cases span several vocab tiles, KV tiles and a ragged tail; the named
workloads run at their full sizes in the same launch configuration as the
bench (sampled sequences where the oracle would take minutes).
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ALPHA = 0.3


@pytest.fixture(scope="module")
def gu():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2505_18629_gb300 import build
    build.build()
    import tests.gpu_util as gu
    return gu


def _wl(**kw):
    from paper_2505_18629_gb300 import synth
    base = synth.Workload("case", B=3, gamma=4, R=5, ctx=(0, 300), H=320, Hq=8, Hkv=2, D=128,
                          V=1000, dtype="bf16", p_argmax=0.7, seed=42)
    return base.replace(**kw)


def _check(gu, wl, alpha=ALPHA, ctx=None, seqs=None, check_attn=True, drafts=None,
           preblended=False):
    from paper_2505_18629_gb300 import rv, synth
    if ctx is not None:
        wl = wl.replace(ctx=(min(ctx), max(ctx)))
    inp = synth.generate(wl)
    if ctx is not None:
        inp.ctx_lens[:] = np.asarray(ctx, np.int32)
    if drafts is None:
        drafts = gu.oracle_drafts(inp, alpha, seqs=seqs)
    h = None
    if preblended:
        h = gu.make_handle(wl)
        rv.rv_set_head_mode(h, rv.RV_HEAD_PREBLENDED)
    gpu = gu.run_gpu(inp, drafts, alpha, h=h)
    if h is not None:
        h.close()
    ref = gu.oracle_step(inp, drafts, alpha, seqs=seqs, with_attn=check_attn,
                         preblended=preblended)
    rep = gu.compare(inp, drafts, alpha, ref, gpu, check_attn=check_attn, seqs=seqs)
    print(f"\n{wl.name}: {rep}")
    return inp, drafts, gpu, ref, rep


# ------------------------------------------------------------------ small cases

def test_tiny_fp32_workload(gu):
    from paper_2505_18629_gb300 import synth
    _check(gu, synth.WORKLOADS["tiny"])


def test_bf16_several_tiles_ragged(gu):
    # V=1000: 8 vocab tiles, last one 104 rows; H=320: 5 k-blocks; ctx 0 / 77 / 300
    _check(gu, _wl(), ctx=[0, 77, 300])


def test_bf16_head_dim_64(gu):
    _check(gu, _wl(D=64, Hq=4, Hkv=4, seed=43), ctx=[5, 129, 64])


def test_bf16_gqa8_two_row_groups(gu):
    # G=8, Lb=20 -> 160 query rows per KV head: two row groups
    _check(gu, _wl(Hq=16, Hkv=2, gamma=6, R=8, B=2, seed=44), ctx=[1000, 3])


def test_bf16_tcgen05_attention_ragged(gu):
    # B*Hkv = 40 (sequence, KV head) pairs selects the tcgen05 attention kernel;
    # ragged contexts, an empty cache, and a context spanning several key tiles
    _check(gu, _wl(B=20, Hq=8, Hkv=2, gamma=3, R=4, V=600, H=256, ctx=(0, 700), seed=60))


def test_bf16_tcgen05_attention_gqa8_two_row_groups(gu):
    # G=8, Lb=20: 160 query rows per KV head -> two 128-row MMA groups
    _check(gu, _wl(B=20, Hq=16, Hkv=2, gamma=6, R=8, V=500, H=128, ctx=(1, 300), seed=61))


def _attention_only(gu, inp, ctx, h):
    """rv_verify_attention alone on fresh cache copies; returns (out bits, status)."""
    import torch
    from paper_2505_18629_gb300 import rv
    q, kb, vb = gu.to_dev(inp.q), gu.to_dev(inp.k_blk), gu.to_dev(inp.v_blk)
    kc, vc = gu.to_dev(inp.k_cache), gu.to_dev(inp.v_cache)
    out = torch.zeros_like(q)
    rv.rv_verify_attention(h, q, kb, vb, kc, vc, gu.to_dev(np.asarray(ctx, np.int32)), out)
    return gu.to_np(out), rv.rv_read_status(h), gu.to_np(kc)


def test_tcgen05_attention_chunk_boundaries_and_repeated_launches(gu):
    # B*Hkv = 40 selects the persistent tcgen05 kernel; its key chunks are 256
    # keys here, so contexts at and around 128 / 256 / 512 / 768 hit tile and
    # chunk edges, and three launches on one handle check that the item
    # counter is re-armed between launches.
    import oracle.rv_oracle as orc
    from paper_2505_18629_gb300 import synth
    wl = _wl(B=20, Hq=8, Hkv=2, gamma=3, R=4, V=600, H=256, ctx=(0, 1200), seed=62)
    inp = synth.generate(wl)
    h = gu.make_handle(wl)
    edges = [0, 1, 127, 128, 255, 256, 257, 511, 512, 513, 767, 768, 769, 1023, 1024, 1100, 2, 64,
             384, wl.capacity - wl.Lb]
    rng = np.random.default_rng(7)
    for rep in range(3):
        ctx = np.asarray(edges if rep == 0 else rng.permutation(edges), np.int32)
        out, status, kc = _attention_only(gu, inp, ctx, h)
        assert status == 0
        ref, rkc, _ = orc.verify_attention(inp.q, inp.k_blk, inp.v_blk, inp.k_cache, inp.v_cache, ctx)
        ok, amax, nbad = gu.attn_close(out, ref)
        assert ok, f"launch {rep}: {nbad} elements beyond tolerance (max {amax:.3g})"
        for b in range(wl.B):
            c = int(ctx[b])
            np.testing.assert_array_equal(kc[b, :, :c + wl.Lb],
                                          gu._bits_like(rkc[b, :, :c + wl.Lb], kc))
    h.close()


def test_tcgen05_attention_context_overflow(gu):
    import oracle.rv_oracle as orc
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(B=20, Hq=8, Hkv=2, gamma=3, R=4, V=600, H=256, ctx=(0, 600), seed=63)
    inp = synth.generate(wl)
    ctx = inp.ctx_lens.astype(np.int32).copy()
    ctx[3] = wl.capacity - wl.Lb + 1                        # does not fit
    ctx[11] = -1                                            # negative
    h = gu.make_handle(wl)
    out, status, kc = _attention_only(gu, inp, ctx, h)
    assert status & rv.RV_DEV_CTX_RANGE
    assert (out[3] == 0).all() and (out[11] == 0).all()     # left untouched
    np.testing.assert_array_equal(kc[3], inp.k_cache[3])
    ok_seqs = [b for b in range(wl.B) if b not in (3, 11)]
    ref, _, _ = orc.verify_attention(inp.q[ok_seqs], inp.k_blk[ok_seqs], inp.v_blk[ok_seqs],
                                     inp.k_cache[ok_seqs], inp.v_cache[ok_seqs], ctx[ok_seqs])
    ok, amax, nbad = gu.attn_close(out[ok_seqs], ref)
    assert ok, f"{nbad} elements beyond tolerance (max {amax:.3g})"
    h.close()


def test_bf16_max_pairs_single_chunk(gu):
    # B*(gamma+1) = 126 pairs -> N = 256 columns, the widest MMA
    _check(gu, _wl(B=14, gamma=8, R=8, V=777, H=256, ctx=(10, 60), seed=45), check_attn=False)


def test_bf16_multi_chunk(gu):
    # 180 pairs -> two chunks of 90 (N = 192 each)
    _check(gu, _wl(B=20, gamma=8, R=2, V=1500, H=128, ctx=(1, 40), seed=46), check_attn=False)


@pytest.mark.parametrize("B,gamma,V", [(16, 8, 1000), (16, 8, 60000), (15, 9, 60000)])
def test_bf16_pair_kernel_two_chunks_many_tiles(gu, B, gamma, V):
    # 144 / 150 pairs in one chunk on CTA pairs, two sub-groups in the split
    # accumulator layout: 32 + 112 pairs / 64 + 96 (160 with 10 padding
    # pairs); at V = 60000 every CTA pair runs several vocab tiles, so the
    # small sub-group's slot is reused every tile, the large one's two by
    # turns, and their barrier phases flip; H = 320 leaves a half-filled last
    # K stage
    _check(gu, _wl(B=B, gamma=gamma, R=3, V=V, H=320, ctx=(1, 30), seed=47 + V % 7),
           check_attn=False)


def test_bf16_no_template_gamma1(gu):
    _check(gu, _wl(gamma=1, R=0, B=2, seed=47), ctx=[3, 0])


def test_alpha_zero_fused_equals_original(gu):
    _, _, gpu, _, _ = _check(gu, _wl(seed=48), alpha=0.0, ctx=[2, 3, 4])
    np.testing.assert_array_equal(gpu.scores[..., 2], gpu.scores[..., 0])
    np.testing.assert_array_equal(gpu.scores[:, :-1, 3], gpu.scores[:, :-1, 4])


def test_alpha_one_fused_equals_reflective(gu):
    _, _, gpu, _, _ = _check(gu, _wl(seed=49), alpha=1.0, ctx=[2, 3, 4])
    np.testing.assert_array_equal(gpu.scores[..., 2], gpu.scores[..., 1])


def test_all_accepted_and_none_accepted(gu):
    from paper_2505_18629_gb300 import synth
    wl = _wl(seed=50, B=2)
    inp = synth.generate(wl)
    inp.ctx_lens[:] = [10, 20]
    choice = gu.oracle_choice(inp, ALPHA).astype(np.int32)
    drafts = choice.copy()
    drafts[1] = (choice[1] + 1) % wl.V                      # every draft of seq 1 is wrong
    gpu = gu.run_gpu(inp, drafts, ALPHA)
    ref = gu.oracle_step(inp, drafts, ALPHA)
    gu.compare(inp, drafts, ALPHA, ref, gpu)
    assert int(ref["accepted_len"][0]) == wl.gamma and int(ref["accepted_len"][1]) == 0


def test_pack_block_entry_point(gu):
    import torch
    import oracle.rv_oracle as orc
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(seed=53, B=3, gamma=5, R=7)
    inp = synth.generate(wl)
    h = gu.make_handle(wl)
    d = gu.to_dev(inp.draft_alt)
    blk = torch.full((3, wl.Lb), -1, dtype=torch.int32, device="cuda")
    pos = torch.full_like(blk, -1)
    rv.rv_pack_block(h, d, gu.to_dev(inp.prompt_ids), gu.to_dev(inp.prefix_ids),
                     gu.to_dev(inp.ctx_lens), blk, pos)
    ref_b, ref_p = orc.pack_block(inp.draft_alt, inp.prompt_ids, inp.prefix_ids, inp.ctx_lens)
    np.testing.assert_array_equal(gu.to_np(blk), ref_b)
    np.testing.assert_array_equal(gu.to_np(pos), ref_p)
    h.close()


def test_separate_entry_points_match_step(gu):
    """rv_verify_attention + rv_verify_head + rv_accept == rv_verify_step."""
    import torch
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(seed=54, B=3)
    inp = synth.generate(wl)
    drafts = gu.oracle_drafts(inp, ALPHA)
    step = gu.run_gpu(inp, drafts, ALPHA)
    h = gu.make_handle(wl)
    g = wl.gamma
    q, kb, vb = gu.to_dev(inp.q), gu.to_dev(inp.k_blk), gu.to_dev(inp.v_blk)
    kc, vc = gu.to_dev(inp.k_cache), gu.to_dev(inp.v_cache)
    ctx, d = gu.to_dev(inp.ctx_lens), gu.to_dev(drafts.astype(np.int32))
    attn = torch.zeros_like(q)
    rv.rv_verify_attention(h, q, kb, vb, kc, vc, ctx, attn)
    sc = torch.empty((wl.B, g + 1, rv.RV_NSCORES), device="cuda")
    am = torch.empty((wl.B, g + 1), dtype=torch.int32, device="cuda")
    mg = torch.empty((wl.B, g), device="cuda")
    rv.rv_verify_head(h, gu.to_dev(inp.hidden), gu.to_dev(inp.W), d, g, wl.R, ALPHA, sc, am, mg)
    acc = torch.empty((wl.B, g), dtype=torch.uint8, device="cuda")
    al = torch.empty((wl.B,), dtype=torch.int32, device="cuda")
    nt, co = torch.empty_like(al), torch.empty_like(al)
    rv.rv_accept(h, d, am, acc, al, nt, ctx, co)
    assert rv.rv_read_status(h) == 0
    np.testing.assert_array_equal(gu.to_np(attn), step.attn)
    # The LM head claims vocab tiles dynamically, so the order in which the
    # per-CTA statistics merge (and their fp32 rounding) varies run to run.
    _same_decisions(gu, gu.to_np(sc), gu.to_np(am), gu.to_np(mg), step)
    np.testing.assert_array_equal(gu.to_np(acc), step.accept_mask)
    np.testing.assert_array_equal(gu.to_np(al), step.accepted_len)
    np.testing.assert_array_equal(gu.to_np(nt), step.next_token)
    np.testing.assert_array_equal(gu.to_np(co), step.ctx_out)
    h.close()


def _same_decisions(gu, scores, argmax, margin, step, atol=1e-4):
    np.testing.assert_allclose(scores, step.scores, atol=atol, rtol=0)
    np.testing.assert_allclose(margin, step.margin, atol=atol, rtol=0)
    clear = np.concatenate([step.margin, np.full((step.margin.shape[0], 1), np.inf)], 1) > atol
    assert ((argmax == step.argmax) | ~clear).all()


def test_host_buffer_step_matches_device_step(gu):
    import torch
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(seed=55, B=2)
    inp = synth.generate(wl)
    drafts = gu.oracle_drafts(inp, ALPHA)
    step = gu.run_gpu(inp, drafts, ALPHA)
    h = gu.make_handle(wl)
    g, B, Lb = wl.gamma, wl.B, wl.Lb

    def host(x):
        t = torch.from_numpy(x.view(np.int16) if x.dtype == np.uint16 else np.ascontiguousarray(x))
        return (t.view(torch.bfloat16) if x.dtype == np.uint16 else t).pin_memory()
    kc, vc = gu.to_dev(inp.k_cache), gu.to_dev(inp.v_cache)
    outs = dict(blk=torch.empty((B, Lb), dtype=torch.int32), pos=torch.empty((B, Lb), dtype=torch.int32),
                attn=torch.empty(inp.q.shape, dtype=torch.bfloat16),
                sc=torch.empty((B, g + 1, rv.RV_NSCORES)), am=torch.empty((B, g + 1), dtype=torch.int32),
                mg=torch.empty((B, g)), acc=torch.empty((B, g), dtype=torch.uint8),
                al=torch.empty((B,), dtype=torch.int32), nt=torch.empty((B,), dtype=torch.int32),
                co=torch.empty((B,), dtype=torch.int32))
    outs = {k: v.pin_memory() for k, v in outs.items()}
    h2d, d2h = rv.rv_verify_step_host(
        h, host(inp.q), host(inp.k_blk), host(inp.v_blk), kc, vc, host(inp.hidden),
        gu.to_dev(inp.W), host(drafts.astype(np.int32)), host(inp.prompt_ids), host(inp.prefix_ids),
        host(inp.ctx_lens), ALPHA, outs["blk"], outs["pos"], outs["attn"], outs["sc"], outs["am"],
        outs["mg"], outs["acc"], outs["al"], outs["nt"], outs["co"])
    assert h2d > 0 and d2h > 0
    np.testing.assert_array_equal(outs["blk"].numpy(), step.block_ids)
    np.testing.assert_array_equal(outs["attn"].view(torch.int16).numpy().view(np.uint16), step.attn)
    _same_decisions(gu, outs["sc"].numpy(), outs["am"].numpy(), outs["mg"].numpy(), step)
    np.testing.assert_array_equal(outs["al"].numpy(), step.accepted_len)
    np.testing.assert_array_equal(outs["nt"].numpy(), step.next_token)
    # the prepared form of the same call, twice on the same buffers (the cache
    # gets the same block appended again at the same positions)
    for v in outs.values():
        v.zero_()
    ins = [host(inp.q), host(inp.k_blk), host(inp.v_blk), kc, vc, host(inp.hidden),
           gu.to_dev(inp.W), host(drafts.astype(np.int32)), host(inp.prompt_ids),
           host(inp.prefix_ids), host(inp.ctx_lens)]
    prep = rv.PreparedStepHost(h, *ins, ALPHA, outs["blk"], outs["pos"], outs["attn"], outs["sc"],
                               outs["am"], outs["mg"], outs["acc"], outs["al"], outs["nt"],
                               outs["co"])
    for _ in range(2):
        assert prep() == (h2d, d2h)
        np.testing.assert_array_equal(outs["blk"].numpy(), step.block_ids)
        np.testing.assert_array_equal(outs["attn"].view(torch.int16).numpy().view(np.uint16),
                                      step.attn)
        _same_decisions(gu, outs["sc"].numpy(), outs["am"].numpy(), outs["mg"].numpy(), step)
        np.testing.assert_array_equal(outs["al"].numpy(), step.accepted_len)
        np.testing.assert_array_equal(outs["co"].numpy(), step.ctx_out)
    h.close()


def test_host_buffer_step_graph_replay(gu):
    # the same call repeated on a non-default stream is captured once as a CUDA
    # graph and replayed; new contents of the pinned inputs (here the drafts)
    # flow through every replay, and the launch count grows as for direct calls
    import torch
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(seed=56, B=2)
    inp = synth.generate(wl)
    d1 = gu.oracle_drafts(inp, ALPHA)
    d2 = ((d1 + 1) % wl.V).astype(d1.dtype)
    ref = {1: gu.run_gpu(inp, d1, ALPHA), 2: gu.run_gpu(inp, d2, ALPHA)}
    h = gu.make_handle(wl)
    g, B, Lb = wl.gamma, wl.B, wl.Lb

    def host(x):
        t = torch.from_numpy(x.view(np.int16) if x.dtype == np.uint16 else np.ascontiguousarray(x))
        return (t.view(torch.bfloat16) if x.dtype == np.uint16 else t).pin_memory()
    kc, vc = gu.to_dev(inp.k_cache), gu.to_dev(inp.v_cache)
    outs = dict(blk=torch.empty((B, Lb), dtype=torch.int32), pos=torch.empty((B, Lb), dtype=torch.int32),
                attn=torch.empty(inp.q.shape, dtype=torch.bfloat16),
                sc=torch.empty((B, g + 1, rv.RV_NSCORES)), am=torch.empty((B, g + 1), dtype=torch.int32),
                mg=torch.empty((B, g)), acc=torch.empty((B, g), dtype=torch.uint8),
                al=torch.empty((B,), dtype=torch.int32), nt=torch.empty((B,), dtype=torch.int32),
                co=torch.empty((B,), dtype=torch.int32))
    outs = {k: v.pin_memory() for k, v in outs.items()}
    drafts = host(d1.astype(np.int32))
    stream = torch.cuda.Stream()
    prep = rv.PreparedStepHost(h, host(inp.q), host(inp.k_blk), host(inp.v_blk), kc, vc,
                               host(inp.hidden), gu.to_dev(inp.W), drafts, host(inp.prompt_ids),
                               host(inp.prefix_ids), host(inp.ctx_lens), ALPHA, outs["blk"],
                               outs["pos"], outs["attn"], outs["sc"], outs["am"], outs["mg"],
                               outs["acc"], outs["al"], outs["nt"], outs["co"], stream)
    counts = []
    for which in (1, 1, 2, 1, 2):
        drafts.copy_(torch.from_numpy((d1 if which == 1 else d2).astype(np.int32)))
        for v in outs.values():
            v.zero_()
        n0 = rv.rv_launch_count(h)
        prep()
        counts.append(rv.rv_launch_count(h) - n0)
        step = ref[which]
        np.testing.assert_array_equal(outs["blk"].numpy(), step.block_ids)
        np.testing.assert_array_equal(outs["attn"].view(torch.int16).numpy().view(np.uint16),
                                      step.attn)
        _same_decisions(gu, outs["sc"].numpy(), outs["am"].numpy(), outs["mg"].numpy(), step)
        np.testing.assert_array_equal(outs["acc"].numpy(), step.accept_mask)
        np.testing.assert_array_equal(outs["al"].numpy(), step.accepted_len)
        np.testing.assert_array_equal(outs["nt"].numpy(), step.next_token)
        np.testing.assert_array_equal(outs["co"].numpy(), step.ctx_out)
    assert len(set(counts)) == 1 and counts[0] > 0, counts
    assert rv.rv_host_step_graphed(h)
    assert rv.rv_read_status(h) == 0
    h.close()


# ------------------------------------------------------------------ device-side checks

def test_out_of_range_draft_sets_status(gu):
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(seed=51, B=2)
    inp = synth.generate(wl)
    inp.ctx_lens[:] = [4, 4]
    drafts = gu.oracle_drafts(inp, ALPHA)
    drafts[0, 1] = wl.V + 5
    gpu = gu.run_gpu(inp, drafts, ALPHA)
    assert gpu.status & rv.RV_DEV_DRAFT_RANGE
    assert gpu.accept_mask[0, 1] == 0 and gpu.accepted_len[0] <= 1
    assert np.isnan(gpu.scores[0, 1, 3]) and np.isnan(gpu.margin[0, 1])


def test_context_overflow_sets_status_and_skips(gu):
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(seed=52, B=2)
    inp = synth.generate(wl)
    inp.ctx_lens[:] = [wl.capacity - wl.Lb + 1, 5]          # seq 0 does not fit
    drafts = gu.oracle_drafts(inp, ALPHA)
    gpu = gu.run_gpu(inp, drafts, ALPHA)
    assert gpu.status & rv.RV_DEV_CTX_RANGE
    assert (gpu.attn[0] == 0).all()                         # left untouched (zeros)
    np.testing.assert_array_equal(gpu.k_cache[0], inp.k_cache[0])


def test_host_validation_errors(gu):
    import torch
    from paper_2505_18629_gb300 import rv
    wl = _wl()
    h = gu.make_handle(wl)
    g, R = wl.gamma, wl.R
    W = torch.zeros((wl.V, wl.H), dtype=torch.bfloat16, device="cuda")

    def head(B, alpha):
        rv.rv_verify_head(h, torch.zeros((B, 2 * g + R + 1, wl.H), dtype=torch.bfloat16,
                                         device="cuda"), W,
                          torch.zeros((B, g), dtype=torch.int32, device="cuda"), g, R, alpha,
                          torch.zeros((B, g + 1, rv.RV_NSCORES), device="cuda"),
                          torch.zeros((B, g + 1), dtype=torch.int32, device="cuda"),
                          torch.zeros((B, g), device="cuda"))
    with pytest.raises(rv.RVError) as e:
        head(4, 0.3)
    assert e.value.code == rv.RV_ERR_CAPACITY                # B=4 > max_batch=3
    with pytest.raises(rv.RVError) as e:
        head(1, float("nan"))
    assert e.value.code == rv.RV_ERR_INVALID_ARG
    # a hidden tensor with too few rows is refused by the binding, before any launch
    with pytest.raises(ValueError, match="hidden"):
        rv.rv_verify_head(h, torch.zeros((1, 2 * g + R, wl.H), dtype=torch.bfloat16,
                                         device="cuda"), W,
                          torch.zeros((1, g), dtype=torch.int32, device="cuda"), g, R, 0.3,
                          torch.zeros((1, g + 1, rv.RV_NSCORES), device="cuda"),
                          torch.zeros((1, g + 1), dtype=torch.int32, device="cuda"),
                          torch.zeros((1, g), device="cuda"))
    h.close()


# ------------------------------------------------------------------ typical acceptance (Alg. 3)

def _typical_params(gu, inp, drafts, alpha, bind):
    """eps / delta that split the drafts about half and half: the entropy term
    binds (bind='delta') or the constant eps does (bind='eps')."""
    ref = gu.oracle_step(inp, drafts, alpha, with_attn=False)
    p = np.exp(ref["logp_fused"])
    if bind == "delta":
        return 1.0, float(np.median(p * np.exp(ref["ent_orig"][:, :-1])))
    return float(np.median(p)), 1e30


@pytest.mark.parametrize("bind", ["delta", "eps"])
def test_typical_acceptance_step(gu, bind):
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(B=6, gamma=5, seed=70)
    inp = synth.generate(wl)
    drafts = gu.oracle_drafts(inp, ALPHA)
    eps, delta = _typical_params(gu, inp, drafts, ALPHA, bind)
    h = gu.make_handle(wl)
    rv.rv_set_acceptance(h, rv.RV_ACCEPT_TYPICAL, eps, delta)
    gpu = gu.run_gpu(inp, drafts, ALPHA, h=h)
    ref = gu.oracle_typical(inp, drafts, ALPHA, eps, delta)
    rep = gu.compare(inp, drafts, ALPHA, ref, gpu)
    assert 0 < ref["accept_mask"].sum() < ref["accept_mask"].size
    print(f"\ntypical ({bind}): {rep}")
    # back to exact match on the same handle
    rv.rv_set_acceptance(h, rv.RV_ACCEPT_EXACT)
    gpu = gu.run_gpu(inp, drafts, ALPHA, h=h)
    gu.compare(inp, drafts, ALPHA, gu.oracle_step(inp, drafts, ALPHA), gpu)
    h.close()


def test_typical_acceptance_separate_entry_points(gu):
    import torch
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(B=5, gamma=4, seed=71)
    inp = synth.generate(wl)
    drafts = gu.oracle_drafts(inp, ALPHA)
    eps, delta = _typical_params(gu, inp, drafts, ALPHA, "delta")
    h = gu.make_handle(wl)
    B, g = wl.B, wl.gamma
    d = gu.to_dev(drafts.astype(np.int32))
    sc = torch.empty((B, g + 1, rv.RV_NSCORES), device="cuda")
    am = torch.empty((B, g + 1), dtype=torch.int32, device="cuda")
    mg = torch.empty((B, g), device="cuda")
    rv.rv_verify_head(h, gu.to_dev(inp.hidden), gu.to_dev(inp.W), d, g, wl.R, ALPHA, sc, am, mg)
    acc = torch.empty((B, g), dtype=torch.uint8, device="cuda")
    n = torch.empty((B,), dtype=torch.int32, device="cuda")
    t = torch.empty_like(n)
    ctx = gu.to_dev(inp.ctx_lens.astype(np.int32))
    co = torch.empty_like(ctx)
    rv.rv_accept_typical(h, d, sc, am, eps, delta, acc, n, t, ctx, co)
    ref = gu.oracle_typical(inp, drafts, ALPHA, eps, delta, with_attn=False)
    low = np.abs(ref["typical_gap"]) < gu.MARGIN_EPS
    assert not ((gu.to_np(acc) != ref["accept_mask"]) & ~low).any()
    if not low.any():
        np.testing.assert_array_equal(gu.to_np(n), ref["accepted_len"])
        np.testing.assert_array_equal(gu.to_np(t), ref["next_token"])
    np.testing.assert_allclose(gu.to_np(sc)[..., rv.RV_SCORE_ENT_ORIG], ref["ent_orig"], atol=gu.LOGP_ATOL)
    with pytest.raises(rv.RVError):
        rv.rv_accept_typical(h, d, sc, am, 0.0, delta, acc, n, t, ctx, co)
    with pytest.raises(rv.RVError):
        rv.rv_set_acceptance(h, 7, 0.1, 0.1)
    h.close()


def test_typical_acceptance_fp32_and_pairs(gu):
    # the fp32 CUDA-core head and the CTA-pair tensor-core head (N >= 96)
    from paper_2505_18629_gb300 import rv, synth
    for wl in (synth.WORKLOADS["tiny"], _wl(B=14, gamma=8, R=8, V=777, H=256, ctx=(10, 60), seed=72)):
        inp = synth.generate(wl)
        drafts = gu.oracle_drafts(inp, ALPHA)
        eps, delta = _typical_params(gu, inp, drafts, ALPHA, "delta")
        h = gu.make_handle(wl)
        rv.rv_set_acceptance(h, rv.RV_ACCEPT_TYPICAL, eps, delta)
        gpu = gu.run_gpu(inp, drafts, ALPHA, h=h)
        ref = gu.oracle_typical(inp, drafts, ALPHA, eps, delta)
        gu.compare(inp, drafts, ALPHA, ref, gpu)
        h.close()


# ------------------------------------------------------------------ speculative sampling (Alg. 1)

SPEC_TOL = 2e-3  # decisions / CDF positions this close to a boundary may differ (fp32 vs fp64)


def _spec_inputs(inp, alpha, seed, same=False):
    """Draft distributions q_i (float32) near the oracle's fused p_i, drafts
    x_i ~ q_i, uniforms r and u; plus the oracle's fused logits z."""
    import oracle.rv_oracle as orc
    wl = inp.wl
    rng = np.random.default_rng(seed)
    dummy = np.zeros((wl.B, wl.gamma), np.int64)
    z = orc.verify_head(inp.W, inp.hidden, dummy, wl.gamma, wl.R, alpha)["z"]
    logit_q = z[:, :wl.gamma] + (0.0 if same else rng.normal(0, 1.0, z[:, :wl.gamma].shape))
    q = np.exp(logit_q - logit_q.max(-1, keepdims=True))
    q = (q / q.sum(-1, keepdims=True)).astype(np.float32)
    q64 = q.astype(np.float64) / q.astype(np.float64).sum(-1, keepdims=True)
    drafts = np.array([[rng.choice(wl.V, p=q64[b, i]) for i in range(wl.gamma)]
                       for b in range(wl.B)], np.int64)
    r = rng.uniform(0, 1, (wl.B, wl.gamma)).astype(np.float32)
    u = rng.uniform(0, 1, wl.B).astype(np.float32)
    return z, q, drafts, r, u


def _run_spec(gu, inp, drafts, alpha, q, r, u, separate=False):
    import torch
    from paper_2505_18629_gb300 import rv
    wl = inp.wl
    B, g = wl.B, wl.gamma
    h = gu.make_handle(wl)
    rv.rv_set_acceptance(h, rv.RV_ACCEPT_SPECULATIVE)
    dq, dr, du = gu.to_dev(q), gu.to_dev(r), gu.to_dev(u)
    d = gu.to_dev(drafts.astype(np.int32))
    ctx = gu.to_dev(inp.ctx_lens.astype(np.int32))
    sc = torch.empty((B, g + 1, rv.RV_NSCORES), device="cuda")
    am = torch.empty((B, g + 1), dtype=torch.int32, device="cuda")
    mg = torch.empty((B, g), device="cuda")
    acc = torch.full((B, g), 7, dtype=torch.uint8, device="cuda")
    n = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    t = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    co = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    if separate:
        rv.rv_verify_head(h, gu.to_dev(inp.hidden), gu.to_dev(inp.W), d, g, wl.R, alpha, sc, am, mg)
        rv.rv_accept_speculative(h, d, dq, dr, du, sc, acc, n, t, ctx, co)
    else:
        q_, kb, vb = gu.to_dev(inp.q), gu.to_dev(inp.k_blk), gu.to_dev(inp.v_blk)
        kc, vc = gu.to_dev(inp.k_cache), gu.to_dev(inp.v_cache)
        prompt = gu.to_dev(inp.prompt_ids.astype(np.int32)) if inp.prompt_ids.size else None
        prefix = gu.to_dev(inp.prefix_ids.astype(np.int32))
        attn = torch.zeros_like(q_)
        with pytest.raises(rv.RVError):  # plain step refuses the sampling rule (no q)
            rv.rv_verify_step(h, q_, kb, vb, kc, vc, gu.to_dev(inp.hidden), gu.to_dev(inp.W), d,
                              prompt, prefix, ctx, alpha, None, None, attn, sc, am, mg, acc, n, t, co)
        rv.rv_verify_step_speculative(h, q_, kb, vb, kc, vc, gu.to_dev(inp.hidden),
                                      gu.to_dev(inp.W), d, prompt, prefix, ctx, alpha, dq, dr, du,
                                      None, None, attn, sc, am, mg, acc, n, t, co)
    status = rv.rv_read_status(h)
    h.close()
    return gu.to_np(acc), gu.to_np(n), gu.to_np(t), gu.to_np(co), gu.to_np(sc), status


def _check_spec(inp, z, q, drafts, r, u, gpu):
    import oracle.rv_oracle as orc
    wl = inp.wl
    g = wl.gamma
    acc_g, n_g, t_g, co_g, sc_g, status = gpu
    assert status == 0
    q64 = q.astype(np.float64) / q.astype(np.float64).sum(-1, keepdims=True)
    acc, n, t, log_ratio, _ = orc.speculative_accept(drafts, z, q64, r.astype(np.float64),
                                                     u.astype(np.float64))
    close = np.abs(np.log(r.astype(np.float64)) - log_ratio) < SPEC_TOL
    assert not ((acc_g.astype(bool) != acc) & ~close).any(), "accept decision differs at a clear case"
    logp = z - orc.logsumexp(z)[..., None]
    p = np.exp(logp)
    n_match = 0
    for b in range(wl.B):
        nb = int(n_g[b])
        assert acc_g[b, :nb].all() and (nb == g or acc_g[b, nb] == 0)
        assert co_g[b] == inp.ctx_lens[b] + nb
        if nb != n[b]:
            assert close[b, :min(n[b], nb) + 1].any(), f"sequence {b}: n {nb} vs {n[b]}"
            continue
        n_match += 1
        w = np.maximum(0.0, p[b, nb] - q64[b, nb]) if nb < g else p[b, nb]
        c = np.cumsum(w) / w.sum()
        tb = int(t_g[b])
        lo = c[tb - 1] if tb > 0 else 0.0
        assert lo - SPEC_TOL <= u[b] <= c[tb] + SPEC_TOL, \
            f"sequence {b}: t {tb} at CDF [{lo:.5f}, {c[tb]:.5f}] for u {u[b]:.5f}"
    assert n_match >= wl.B // 2
    return acc, n


@pytest.mark.parametrize("separate", [False, True])
def test_speculative_sampling_small(gu, separate):
    from paper_2505_18629_gb300 import synth
    wl = _wl(B=8, gamma=5, V=1000, seed=80)
    inp = synth.generate(wl)
    z, q, drafts, r, u = _spec_inputs(inp, ALPHA, 81)
    acc, n = _check_spec(inp, z, q, drafts, r, u,
                         _run_spec(gu, inp, drafts, ALPHA, q, r, u, separate=separate))
    assert 0 < acc.sum() < acc.size


def test_speculative_sampling_draft_equals_target(gu):
    # q = p (up to float32): every draft is kept and t ~ p_{gamma+1}
    from paper_2505_18629_gb300 import synth
    wl = _wl(B=6, gamma=4, V=1000, seed=82)
    inp = synth.generate(wl)
    z, q, drafts, r, u = _spec_inputs(inp, ALPHA, 83, same=True)
    r = np.minimum(r, 0.99).astype(np.float32)
    acc, n = _check_spec(inp, z, q, drafts, r, u, _run_spec(gu, inp, drafts, ALPHA, q, r, u))
    assert acc.all()


def test_speculative_sampling_pairs_and_8b(gu):
    # the CTA-pair head (N >= 96) and the full 8B batch-1 vocabulary
    from paper_2505_18629_gb300 import synth
    for wl, seqs_ok in ((_wl(B=14, gamma=8, R=8, V=777, H=256, ctx=(10, 60), seed=84), None),
                        (synth.WORKLOADS["llama3-8b-b1"], None)):
        inp = synth.generate(wl)
        z, q, drafts, r, u = _spec_inputs(inp, ALPHA, 85)
        _check_spec(inp, z, q, drafts, r, u, _run_spec(gu, inp, drafts, ALPHA, q, r, u))


# ------------------------------------------------------------------ sampled exact match (Alg. 2, temperature T)

def _sampled_inputs(inp, alpha, T, seed, keep=0.7, preblended=False):
    """The oracle's fused logits z, uniforms u [B, gamma+1], and drafts that
    equal the oracle's sampled target token with probability `keep`."""
    import oracle.rv_oracle as orc
    wl = inp.wl
    rng = np.random.default_rng(seed)
    dummy = np.zeros((wl.B, wl.gamma), np.int64)
    head_fn = orc.verify_head_preblended if preblended else orc.verify_head
    z = head_fn(inp.W, inp.hidden, dummy, wl.gamma, wl.R, alpha)["z"]
    u = rng.uniform(0, 1, (wl.B, wl.gamma + 1)).astype(np.float32)
    _, _, _, xhat, _ = orc.sampled_exact_accept(dummy, z, T, u.astype(np.float64))
    alt = rng.integers(0, wl.V, (wl.B, wl.gamma))
    drafts = np.where(rng.uniform(size=(wl.B, wl.gamma)) < keep, xhat[:, :wl.gamma], alt)
    return z, u, drafts.astype(np.int64)


def _run_sampled(gu, inp, drafts, alpha, T, u, separate=False, preblended=False, typical=None):
    """`typical`: (eps, delta) of typical acceptance with t sampled at T."""
    import torch
    from paper_2505_18629_gb300 import rv
    wl = inp.wl
    B, g = wl.B, wl.gamma
    h = gu.make_handle(wl)
    if typical is not None:
        rv.rv_set_acceptance(h, rv.RV_ACCEPT_TYPICAL_SAMPLED, *typical)
    else:
        rv.rv_set_acceptance(h, rv.RV_ACCEPT_SAMPLED)
    if preblended:
        rv.rv_set_head_mode(h, rv.RV_HEAD_PREBLENDED)
    du = gu.to_dev(u)
    d = gu.to_dev(drafts.astype(np.int32))
    ctx = gu.to_dev(inp.ctx_lens.astype(np.int32))
    sc = torch.empty((B, g + 1, rv.RV_NSCORES), device="cuda")
    am = torch.empty((B, g + 1), dtype=torch.int32, device="cuda")
    mg = torch.empty((B, g), device="cuda")
    xs = torch.full((B, g + 1), -7, dtype=torch.int32, device="cuda")
    acc = torch.full((B, g), 7, dtype=torch.uint8, device="cuda")
    n = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    t = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    co = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    if separate:
        rv.rv_verify_head(h, gu.to_dev(inp.hidden), gu.to_dev(inp.W), d, g, wl.R, alpha, sc, am, mg)
        rv.rv_accept_sampled(h, d, du, T, xs, acc, n, t, ctx, co)
    else:
        q_, kb, vb = gu.to_dev(inp.q), gu.to_dev(inp.k_blk), gu.to_dev(inp.v_blk)
        kc, vc = gu.to_dev(inp.k_cache), gu.to_dev(inp.v_cache)
        prompt = gu.to_dev(inp.prompt_ids.astype(np.int32)) if inp.prompt_ids.size else None
        prefix = gu.to_dev(inp.prefix_ids.astype(np.int32))
        attn = torch.zeros_like(q_)
        with pytest.raises(rv.RVError):  # the plain step refuses the sampling rule (no uniforms)
            rv.rv_verify_step(h, q_, kb, vb, kc, vc, gu.to_dev(inp.hidden), gu.to_dev(inp.W), d,
                              prompt, prefix, ctx, alpha, None, None, attn, sc, am, mg, acc, n, t, co)
        with pytest.raises(rv.RVError):  # temperature must be > 0
            rv.rv_verify_step_sampled(h, q_, kb, vb, kc, vc, gu.to_dev(inp.hidden),
                                      gu.to_dev(inp.W), d, prompt, prefix, ctx, alpha, 0.0, du,
                                      None, None, attn, sc, am, mg, xs, acc, n, t, co)
        rv.rv_verify_step_sampled(h, q_, kb, vb, kc, vc, gu.to_dev(inp.hidden), gu.to_dev(inp.W),
                                  d, prompt, prefix, ctx, alpha, T, du, None, None, attn, sc, am,
                                  mg, xs, acc, n, t, co)
    status = rv.rv_read_status(h)
    h.close()
    return (gu.to_np(xs), gu.to_np(acc), gu.to_np(n), gu.to_np(t), gu.to_np(co), gu.to_np(am),
            status)


def _check_sampled(inp, z, u, drafts, T, gpu, min_match=0.9, tol=SPEC_TOL):
    """Sampled tokens equal the oracle's draw except where u lies within
    SPEC_TOL of a cumulative-weight boundary (then the token must be one whose
    CDF interval holds u up to SPEC_TOL); acceptance, n, t and ctx follow the
    GPU's own draws exactly (Alg. 2), and equal the oracle's wherever every
    draw up to n+1 matched."""
    import oracle.rv_oracle as orc
    wl = inp.wl
    g = wl.gamma
    xs, acc, n, t, co, _, status = gpu
    assert status == 0
    acc_o, n_o, t_o, xhat_o, gap = orc.sampled_exact_accept(drafts, z, T, u.astype(np.float64))
    zt = z / T
    p_t = np.exp(zt - orc.logsumexp(zt)[..., None])
    same = xs == xhat_o
    for b, i in zip(*np.nonzero(~same)):
        assert gap[b, i] < tol, f"draw ({b},{i}): {xs[b, i]} vs {xhat_o[b, i]}, gap {gap[b, i]:.2e}"
        c = np.cumsum(p_t[b, i])
        k = int(xs[b, i])
        lo = c[k - 1] if k > 0 else 0.0
        assert lo - tol <= u[b, i] <= c[k] + tol
    assert same.mean() >= min_match, f"only {same.mean():.3f} of the draws match"
    # Alg. 2 on the GPU's own draws: bit-exact
    acc_s, n_s, t_s = orc.exact_match_accept(drafts, xs)
    assert (acc == acc_s).all() and (n == n_s).all() and (t == t_s).all()
    assert (co == inp.ctx_lens + n).all()
    rows_same = same.all(axis=1)
    assert (n[rows_same] == n_o[rows_same]).all() and (t[rows_same] == t_o[rows_same]).all()
    return acc, n


@pytest.mark.parametrize("T,separate", [(1.0, False), (0.8, True), (0.2, False)])
def test_sampled_exact_match_small(gu, T, separate):
    from paper_2505_18629_gb300 import synth
    wl = _wl(B=8, gamma=5, V=1000, seed=90)
    inp = synth.generate(wl)
    z, u, drafts = _sampled_inputs(inp, ALPHA, T, 91)
    acc, n = _check_sampled(inp, z, u, drafts, T,
                            _run_sampled(gu, inp, drafts, ALPHA, T, u, separate=separate))
    assert 0 < acc.sum() < acc.size


def test_sampled_exact_match_low_temperature_is_greedy(gu):
    # T -> 0: every draw is the greedy choice of the head (away from ties)
    from paper_2505_18629_gb300 import synth
    wl = _wl(B=6, gamma=4, V=1500, seed=92)
    inp = synth.generate(wl)
    T = 1e-4
    z, u, drafts = _sampled_inputs(inp, ALPHA, T, 93)
    gpu = _run_sampled(gu, inp, drafts, ALPHA, T, u)
    _check_sampled(inp, z, u, drafts, T, gpu)
    xs, am = gpu[0], gpu[5]
    srt = np.sort(z, axis=-1)
    clear = (srt[..., -1] - srt[..., -2]) > 1e-3
    assert (xs[clear] == am[clear]).all()


@pytest.mark.parametrize("name", ["tiny", "pairs", "llama3-8b-b1"])
def test_sampled_exact_match_kernels_and_8b(gu, name):
    # the fp32 head, the CTA-pair head (N >= 96) and the full 8B vocabulary
    from paper_2505_18629_gb300 import synth
    wl = (_wl(B=14, gamma=8, R=8, V=777, H=256, ctx=(10, 60), seed=94) if name == "pairs"
          else synth.WORKLOADS[name])
    inp = synth.generate(wl)
    z, u, drafts = _sampled_inputs(inp, ALPHA, 0.8, 95)
    gpu = _run_sampled(gu, inp, drafts, ALPHA, 0.8, u)
    if name == "llama3-8b-b1":
        # 128256 tokens: adjacent CDF boundaries are ~1e-5 apart, as close as the
        # fp32-vs-fp64 logit error moves them; a draw may land on a neighbour,
        # whose interval must then hold u within 2e-4
        _check_sampled(inp, z, u, drafts, 0.8, gpu, min_match=0.0, tol=2e-4)
    else:
        _check_sampled(inp, z, u, drafts, 0.8, gpu)


@pytest.mark.parametrize("name", ["pairs-two-subgroups", "pairs-two-chunks", "preblended-two-chunks"])
def test_sampled_exact_match_subtile_draw_layouts(gu, name):
    # inside rv_verify_step_sampled the head leaves per-32-row subtile sums and
    # the draw recomputes one subtile from the head's operands: one chunk of
    # 150 pairs in two sub-groups, two chunks of 160 pairs in two sub-groups,
    # and the pre-blended head over two chunks; vocabularies not a multiple
    # of 32, two temperatures
    pre = name.startswith("preblended")
    B, g = (15, 9) if name == "pairs-two-subgroups" else (32, 9) if not pre else (40, 7)
    V = {"pairs-two-subgroups": 1777, "pairs-two-chunks": 1501, "preblended-two-chunks": 1243}[name]
    from paper_2505_18629_gb300 import synth
    wl = _wl(B=B, gamma=g, R=6, V=V, H=256, ctx=(5, 40), seed=96)
    inp = synth.generate(wl)
    for T in (0.8, 0.3):
        z, u, drafts = _sampled_inputs(inp, ALPHA, T, 97, preblended=pre)
        _check_sampled(inp, z, u, drafts, T, _run_sampled(gu, inp, drafts, ALPHA, T, u,
                                                           preblended=pre))


@pytest.mark.parametrize("name,T", [("small", 0.8), ("pairs", 0.3), ("tiny", 1.0)])
def test_typical_acceptance_sampled_t(gu, name, T):
    # Alg. 3 with t ~ p_{n+1} at temperature T (rv_verify_step_sampled on a
    # handle in RV_ACCEPT_TYPICAL_SAMPLED mode): the one-CTA head, the CTA-pair
    # head and the fp32 head (which writes the fused logits)
    import oracle.rv_oracle as orc
    from paper_2505_18629_gb300 import synth
    wl = {"small": _wl(B=6, gamma=5, seed=73),
          "pairs": _wl(B=14, gamma=8, R=8, V=777, H=256, ctx=(10, 60), seed=74),
          "tiny": synth.WORKLOADS["tiny"]}[name]
    inp = synth.generate(wl)
    drafts = gu.oracle_drafts(inp, ALPHA)
    eps, delta = _typical_params(gu, inp, drafts, ALPHA, "delta")
    head = orc.verify_head(inp.W, inp.hidden, drafts, wl.gamma, wl.R, ALPHA)
    u = np.random.default_rng(75).uniform(0, 1, (wl.B, wl.gamma + 1)).astype(np.float32)
    acc_o, n_o, t_o, gap, cdf_gap = orc.typical_accept_sampled(
        drafts, head["logp_fused"], head["ent_orig"], head["z"], eps, delta, T,
        u.astype(np.float64))
    xs, acc, n, t, co, _, status = _run_sampled(gu, inp, drafts, ALPHA, T, u,
                                                typical=(eps, delta))
    assert status == 0
    low = np.abs(gap) < gu.MARGIN_EPS
    assert not ((acc != acc_o) & ~low).any()
    # n follows the GPU's own mask; t is the GPU's own draw at n+1
    for b in range(wl.B):
        nb = wl.gamma
        for i in range(wl.gamma):
            if not acc[b, i]:
                nb = i
                break
        assert n[b] == nb and t[b] == xs[b, n[b]] and co[b] == inp.ctx_lens[b] + n[b]
    same = (n == n_o)
    assert same.mean() >= 0.5
    # where n agrees, t is the oracle's draw unless u[b, n] sits on a CDF boundary
    for b in np.flatnonzero(same):
        if t[b] != t_o[b]:
            assert cdf_gap[b] < SPEC_TOL, f"sequence {b}: t {t[b]} vs {t_o[b]}"
    assert 0 < acc_o.sum() < acc_o.size


# ------------------------------------------------------------------ pending-token block

def _pending_run(gu, wl, alpha=ALPHA, seed=0, check_attn=True):
    """rv_verify_step_pending against the oracle's verify_step_pending.  The
    workload's block gets one more position in front (the pending token's
    query / key / value, drawn like the others); hidden row 0 is the pending
    token's state, so the head's inputs are the workload's unchanged."""
    import torch
    import oracle.rv_oracle as orc
    from paper_2505_18629_gb300 import rv, synth
    wl = wl.replace(cmax=wl.ctx[1] + wl.Lb + 1)
    inp = synth.generate(wl)
    rng = np.random.default_rng(seed)
    bf = wl.dtype == "bf16"
    std = 1.0 if bf else 0.02

    def front(x):
        row = rng.normal(0, std, x[:, :1].shape).astype(np.float32)
        return np.concatenate([synth.to_bf16_bits(row) if bf else row, x], axis=1)
    inp.q, inp.k_blk, inp.v_blk = front(inp.q), front(inp.k_blk), front(inp.v_blk)
    pending = rng.integers(0, wl.V, wl.B)
    drafts = gu.oracle_drafts(inp, alpha)
    ref = orc.verify_step_pending(inp.W, inp.hidden, inp.q, inp.k_blk, inp.v_blk, inp.k_cache,
                                  inp.v_cache, inp.ctx_lens, pending, drafts, inp.prompt_ids,
                                  inp.prefix_ids, wl.gamma, wl.R, alpha)
    ref.pop("z")
    B, g, Lp = wl.B, wl.gamma, wl.Lb + 1
    h = gu.make_handle(wl)
    W, hidden = gu.to_dev(inp.W), gu.to_dev(inp.hidden)
    q, kb, vb = gu.to_dev(inp.q), gu.to_dev(inp.k_blk), gu.to_dev(inp.v_blk)
    kc, vc = gu.to_dev(inp.k_cache), gu.to_dev(inp.v_cache)
    ctx = gu.to_dev(inp.ctx_lens.astype(np.int32))
    d = gu.to_dev(drafts.astype(np.int32))
    pend = gu.to_dev(pending.astype(np.int32))
    prompt = gu.to_dev(inp.prompt_ids.astype(np.int32)) if inp.prompt_ids.size else None
    prefix = gu.to_dev(inp.prefix_ids.astype(np.int32))
    i32 = dict(dtype=torch.int32, device="cuda")
    block, pos = torch.full((B, Lp), -7, **i32), torch.full((B, Lp), -7, **i32)
    attn = torch.zeros_like(q)
    scores = torch.full((B, g + 1, rv.RV_NSCORES), float("nan"), device="cuda")
    argmax = torch.full((B, g + 1), -7, **i32)
    margin = torch.full((B, g), float("nan"), device="cuda")
    acc = torch.full((B, g), 7, dtype=torch.uint8, device="cuda")
    alen, nxt, co = (torch.full((B,), -7, **i32) for _ in range(3))
    rv.rv_verify_step_pending(h, q, kb, vb, kc, vc, hidden, W, pend, d, prompt, prefix, ctx, alpha,
                              block, pos, attn, scores, argmax, margin, acc, alen, nxt, co)
    status = rv.rv_read_status(h)
    # the separate packing entry point gives the same block
    block2, pos2 = torch.full((B, Lp), -7, **i32), torch.full((B, Lp), -7, **i32)
    rv.rv_pack_block_pending(h, pend, d, prompt, prefix, ctx, block2, pos2)
    torch.cuda.synchronize()
    h.close()
    gpu = gu.GpuRun(gu.to_np(attn), gu.to_np(kc), gu.to_np(vc), gu.to_np(scores),
                    gu.to_np(argmax), gu.to_np(margin), gu.to_np(acc), gu.to_np(alen),
                    gu.to_np(nxt), gu.to_np(co), gu.to_np(block), gu.to_np(pos), status)
    np.testing.assert_array_equal(gu.to_np(block2), gpu.block_ids)
    np.testing.assert_array_equal(gu.to_np(pos2), gpu.pos_ids)
    rep = gu.compare(inp, drafts, alpha, ref, gpu, check_attn=check_attn, pending=pending)
    print(f"\n{wl.name} (pending token): {rep}")
    return rep


@pytest.mark.parametrize("kind", ["mma_sync", "tcgen05", "f32"])
def test_pending_token_step(gu, kind):
    # the small-batch attention (cluster split-KV), the persistent tcgen05
    # attention (B * Hkv = 40), and the fp32 path
    from paper_2505_18629_gb300 import synth
    if kind == "mma_sync":
        wl = _wl(seed=100)
    elif kind == "tcgen05":
        wl = _wl(B=20, Hq=8, Hkv=2, gamma=3, R=4, V=600, H=256, ctx=(0, 700), seed=101)
    else:
        wl = synth.WORKLOADS["tiny"]
    _pending_run(gu, wl, seed=102)


def test_pending_token_step_8b_b16(gu):
    from paper_2505_18629_gb300 import synth
    _pending_run(gu, synth.WORKLOADS["llama3-8b-b16"], seed=103)


# ------------------------------------------------------------------ pre-blended head

@pytest.mark.parametrize("shape", ["ragged", "one-pair", "pairs-144", "two-chunks"])
def test_preblended_head(gu, shape):
    # the head on b_i = bf16(fl((1-a) h) + fl(a h')) against the oracle's
    # verify_head_preblended (whose blend is that rounding, so the tolerance is
    # the plain head's): N = 16 on single CTAs; 144 pairs in one chunk on CTA
    # pairs (above the 128 pairs of a two-distribution chunk); 288 pairs in two
    # chunks of 144 with several vocab tiles per CTA pair
    if shape == "ragged":
        _check(gu, _wl(seed=110), ctx=[0, 77, 300], preblended=True)
    elif shape == "one-pair":
        _check(gu, _wl(B=1, gamma=2, R=4, seed=111), ctx=[5], preblended=True)
    elif shape == "pairs-144":
        _check(gu, _wl(B=16, gamma=8, R=3, V=60000, H=320, ctx=(1, 30), seed=112),
               check_attn=False, preblended=True)
    else:
        _check(gu, _wl(B=32, gamma=8, R=2, V=5000, H=192, ctx=(1, 20), seed=113),
               check_attn=False, preblended=True)


def test_preblended_head_differs_from_fused_by_the_blend_rounding(gu):
    # same inputs through both head modes: the fused-logit statistics agree
    # within the bound of the blend's bf16 rounding, and not bit for bit
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(B=4, gamma=5, V=3000, seed=114)
    inp = synth.generate(wl)
    drafts = gu.oracle_drafts(inp, ALPHA)
    fused = gu.run_gpu(inp, drafts, ALPHA)
    h = gu.make_handle(wl)
    rv.rv_set_head_mode(h, rv.RV_HEAD_PREBLENDED)
    pre = gu.run_gpu(inp, drafts, ALPHA, h=h)
    h.close()
    import oracle.rv_oracle as orc
    d = np.abs(pre.scores[..., 2].astype(np.float64) - fused.scores[..., 2])
    # |dz_v| <= u sum_k |W_vk| |b_k| with u = 2^-8, the bf16 unit roundoff, and
    # |d lse| <= max_v |dz_v|; 1e-4 for the two heads' float32 accumulations
    b = orc.preblend_rows(inp.hidden, wl.gamma, wl.R, ALPHA).astype(np.float64)
    bound = 2.0 ** -8 * (np.abs(b) @ np.abs(orc.as_f64(inp.W)).T).max(axis=-1) + 1e-4
    assert (d <= bound).all()
    assert d.max() > 0
    assert np.isnan(pre.scores[..., [0, 1, 6]]).all()
    assert np.isfinite(fused.scores[..., [0, 1, 6]]).all()


def test_preblended_mode_validation(gu):
    from paper_2505_18629_gb300 import rv, synth
    h = gu.make_handle(_wl())
    with pytest.raises(rv.RVError):
        rv.rv_set_head_mode(h, 7)
    rv.rv_set_acceptance(h, rv.RV_ACCEPT_TYPICAL, 0.3, 0.09)
    with pytest.raises(rv.RVError):  # the typical rule needs the original entropy
        rv.rv_set_head_mode(h, rv.RV_HEAD_PREBLENDED)
    rv.rv_set_acceptance(h, rv.RV_ACCEPT_EXACT)
    rv.rv_set_head_mode(h, rv.RV_HEAD_PREBLENDED)
    with pytest.raises(rv.RVError):
        rv.rv_set_acceptance(h, rv.RV_ACCEPT_TYPICAL, 0.3, 0.09)
    rv.rv_set_head_mode(h, rv.RV_HEAD_FUSED_LOGITS)
    rv.rv_set_acceptance(h, rv.RV_ACCEPT_TYPICAL, 0.3, 0.09)
    h.close()
    h32 = gu.make_handle(synth.WORKLOADS["tiny"])
    with pytest.raises(rv.RVError):  # the bf16 head's variant only
        rv.rv_set_head_mode(h32, rv.RV_HEAD_PREBLENDED)
    h32.close()


@pytest.mark.parametrize("name", ["small", "pairs"])
def test_preblended_sampled_exact_match(gu, name):
    # the pre-blended head writes z for the sampling rule as well
    from paper_2505_18629_gb300 import synth
    wl = (_wl(B=8, gamma=5, V=1000, seed=115) if name == "small"
          else _wl(B=14, gamma=8, R=8, V=777, H=256, ctx=(10, 60), seed=116))
    inp = synth.generate(wl)
    z, u, drafts = _sampled_inputs(inp, ALPHA, 0.8, 117, preblended=True)
    gpu = _run_sampled(gu, inp, drafts, ALPHA, 0.8, u, preblended=True)
    _check_sampled(inp, z, u, drafts, 0.8, gpu)


@pytest.mark.parametrize("name", ["llama3-8b-b1", "llama3-8b-b16"])
def test_preblended_llama3_8b(gu, name):
    from paper_2505_18629_gb300 import synth
    _check(gu, synth.WORKLOADS[name], check_attn=False, preblended=True)


# ------------------------------------------------------------------ standard verification (the baseline)

def _standard_run(gu, wl, seqs=None, check_attn=True, pending=False, host=False):
    """rv_verify_step (or the pending / host-buffer step) of a standard-verification
    handle on the workload's first gamma block positions and gamma+1 hidden rows,
    against the oracle's verify_step_standard."""
    import torch
    import oracle.rv_oracle as orc
    from paper_2505_18629_gb300 import rv, synth
    inp = synth.generate(wl)
    B, g = wl.B, wl.gamma
    S = np.arange(B) if seqs is None else np.asarray(seqs)
    lead = 1 if pending else 0
    hid = np.ascontiguousarray(inp.hidden[:, :g + 1])
    choice = inp.draft_alt.copy()
    choice[S] = orc.verify_head_standard(inp.W, hid[S], np.zeros((len(S), g), np.int64),
                                         g)["argmax"][:, :g]
    drafts = synth.make_drafts(inp, choice)
    t = np.random.default_rng(wl.seed + 7).integers(0, wl.V, B).astype(np.int32)
    Lb = g + lead
    qs, kbs, vbs = (np.ascontiguousarray(x[:, :Lb]) for x in (inp.q, inp.k_blk, inp.v_blk))
    h = gu.make_handle(wl)
    rv.rv_set_head_mode(h, rv.RV_HEAD_STANDARD)
    kc, vc = gu.to_dev(inp.k_cache), gu.to_dev(inp.v_cache)
    W = gu.to_dev(inp.W)
    if host:
        def pin(x):
            tt = torch.from_numpy(x.view(np.int16) if x.dtype == np.uint16 else np.ascontiguousarray(x))
            return (tt.view(torch.bfloat16) if x.dtype == np.uint16 else tt).pin_memory()
        dev = dict(q=pin(qs), kb=pin(kbs), vb=pin(vbs), hid=pin(hid),
                   d=pin(drafts.astype(np.int32)), ctx=pin(inp.ctx_lens.astype(np.int32)))
        mk = lambda shape, dt=torch.int32: torch.full(shape, -7, dtype=dt).pin_memory()
        attn = torch.zeros(qs.shape, dtype=torch.bfloat16).pin_memory()
        sc = torch.full((B, g + 1, rv.RV_NSCORES), float("nan")).pin_memory()
        mg = torch.full((B, g), float("nan")).pin_memory()
    else:
        dev = dict(q=gu.to_dev(qs), kb=gu.to_dev(kbs), vb=gu.to_dev(vbs), hid=gu.to_dev(hid),
                   d=gu.to_dev(drafts.astype(np.int32)), ctx=gu.to_dev(inp.ctx_lens.astype(np.int32)))
        mk = lambda shape, dt=torch.int32: torch.full(shape, -7, dtype=dt, device="cuda")
        attn = torch.zeros_like(dev["q"])
        sc = torch.full((B, g + 1, rv.RV_NSCORES), float("nan"), device="cuda")
        mg = torch.full((B, g), float("nan"), device="cuda")
    prefix = mk((B, 0))
    block, pos = mk((B, Lb)), mk((B, Lb))
    am, acc = mk((B, g + 1)), mk((B, g), torch.uint8)
    n, nt, co = mk((B,)), mk((B,)), mk((B,))
    args = (dev["q"], dev["kb"], dev["vb"], kc, vc, dev["hid"], W)
    tail = (None, prefix, dev["ctx"], ALPHA, block, pos, attn, sc, am, mg, acc, n, nt, co)
    if inp.prompt_ids.size:
        with pytest.raises(rv.RVError):  # standard verification has no template
            prompt = inp.prompt_ids.astype(np.int32)
            if host:
                rv.rv_verify_step_host(h, *args, dev["d"], torch.from_numpy(prompt).pin_memory(),
                                       *tail[1:])
            elif pending:
                rv.rv_verify_step_pending(h, *args, gu.to_dev(t), dev["d"], gu.to_dev(prompt),
                                          *tail[1:])
            else:
                rv.rv_verify_step(h, *args, dev["d"], gu.to_dev(prompt), *tail[1:])
    if host:
        rv.rv_verify_step_host(h, *args, dev["d"], *tail)
    elif pending:
        rv.rv_verify_step_pending(h, *args, gu.to_dev(t), dev["d"], *tail)
    else:
        rv.rv_verify_step(h, *args, dev["d"], *tail)
    torch.cuda.synchronize()
    gpu = gu.GpuRun(gu.to_np(attn), gu.to_np(kc), gu.to_np(vc), gu.to_np(sc), gu.to_np(am),
                    gu.to_np(mg), gu.to_np(acc), gu.to_np(n), gu.to_np(nt), gu.to_np(co),
                    gu.to_np(block), gu.to_np(pos), rv.rv_read_status(h))
    h.close()
    ref = orc.verify_step_standard(inp.W, hid[S], qs[S], kbs[S], vbs[S], inp.k_cache[S],
                                   inp.v_cache[S], inp.ctx_lens[S], drafts[S], g)
    ref.pop("z")
    ref.pop("ctx_out")
    if not check_attn:
        for k in ("attn", "k_cache", "v_cache"):
            ref.pop(k)
    rep = gu.compare(inp, drafts, ALPHA, ref, gpu, check_attn=check_attn, seqs=seqs,
                     pending=t if pending else None, standard=True)
    print(f"\nstandard {wl.name}: {rep}")
    return gpu


def test_standard_verification_small(gu):
    _standard_run(gu, _wl(seed=120), check_attn=True)


def test_standard_verification_tcgen05_attention(gu):
    # B*Hkv = 40 (sequence, KV head) pairs: the persistent tcgen05 attention,
    # here over gamma = 6 block positions
    _standard_run(gu, _wl(B=20, gamma=6, R=8, Hq=16, Hkv=2, V=2000, ctx=(0, 700), seed=121))


def test_standard_verification_pending_block(gu):
    # block [t, x_1..x_gamma]: t's state in hidden row 0, ctx += 1 + n
    _standard_run(gu, _wl(B=3, gamma=4, seed=122), pending=True)


def test_standard_verification_host_buffers(gu):
    _standard_run(gu, _wl(B=4, gamma=5, seed=123), host=True)


# 8B B=16: CTA-pair z-only head (144 pairs); sweep-b16-g4: one-CTA z-only head
# with its merge in a separate launch (80 pairs); sweep-b64-g8: three chunks of
# 192 pairs on CTA pairs.
@pytest.mark.parametrize("name,seqs", [("llama3-8b-b16", None), ("sweep-b16-g4-c1024", [0, 7, 15]),
                                       ("sweep-b64-g8-c8192", [0, 33, 63])])
def test_standard_verification_8b(gu, name, seqs):
    from paper_2505_18629_gb300 import synth
    _standard_run(gu, synth.workload(name), seqs=seqs)


def test_standard_verification_sampled_exact_match(gu):
    # standard verification's head writes z = o for the sampling rule too:
    # rv_verify_head (R = 0, hidden [B, gamma+1, H]) + rv_accept_sampled
    import torch
    import oracle.rv_oracle as orc
    from paper_2505_18629_gb300 import rv, synth
    wl = _wl(B=8, gamma=5, V=1000, seed=124)
    inp = synth.generate(wl)
    B, g, T = wl.B, wl.gamma, 0.8
    hid = np.ascontiguousarray(inp.hidden[:, :g + 1])
    dummy = np.zeros((B, g), np.int64)
    z = orc.verify_head_standard(inp.W, hid, dummy, g)["z"]
    rng = np.random.default_rng(125)
    u = rng.uniform(0, 1, (B, g + 1)).astype(np.float32)
    _, _, _, xhat, _ = orc.sampled_exact_accept(dummy, z, T, u.astype(np.float64))
    drafts = np.where(rng.uniform(size=(B, g)) < 0.7, xhat[:, :g],
                      rng.integers(0, wl.V, (B, g))).astype(np.int64)
    h = gu.make_handle(wl)
    rv.rv_set_head_mode(h, rv.RV_HEAD_STANDARD)
    rv.rv_set_acceptance(h, rv.RV_ACCEPT_SAMPLED)
    d = gu.to_dev(drafts.astype(np.int32))
    ctx = gu.to_dev(inp.ctx_lens.astype(np.int32))
    sc = torch.empty((B, g + 1, rv.RV_NSCORES), device="cuda")
    am = torch.empty((B, g + 1), dtype=torch.int32, device="cuda")
    mg = torch.empty((B, g), device="cuda")
    xs = torch.full((B, g + 1), -7, dtype=torch.int32, device="cuda")
    acc = torch.full((B, g), 7, dtype=torch.uint8, device="cuda")
    n = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    t = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    co = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    with pytest.raises(rv.RVError):  # a template with standard verification
        rv.rv_verify_head(h, gu.to_dev(hid), gu.to_dev(inp.W), d, g, 2, ALPHA, sc, am, mg)
    rv.rv_verify_head(h, gu.to_dev(hid), gu.to_dev(inp.W), d, g, 0, ALPHA, sc, am, mg)
    rv.rv_accept_sampled(h, d, gu.to_dev(u), T, xs, acc, n, t, ctx, co)
    gpu = (gu.to_np(xs), gu.to_np(acc), gu.to_np(n), gu.to_np(t), gu.to_np(co), gu.to_np(am),
           rv.rv_read_status(h))
    h.close()
    acc_np, _ = _check_sampled(inp, z, u, drafts, T, gpu)
    assert 0 < acc_np.sum() < acc_np.size


def test_standard_pack_entry_points(gu):
    import torch
    import oracle.rv_oracle as orc
    from paper_2505_18629_gb300 import rv
    h = gu.make_handle(_wl())
    rv.rv_set_head_mode(h, rv.RV_HEAD_STANDARD)
    d = np.array([[3, 4, 5, 6], [7, 8, 9, 10]], np.int32)
    ctx = np.array([11, 0], np.int32)
    blk = torch.full((2, 5), -7, dtype=torch.int32, device="cuda")
    pos = torch.full((2, 5), -7, dtype=torch.int32, device="cuda")
    empty = torch.zeros((2, 0), dtype=torch.int32, device="cuda")
    b4, p4 = torch.full((2, 4), -7, dtype=torch.int32, device="cuda"), torch.full((2, 4), -7, dtype=torch.int32, device="cuda")
    rv.rv_pack_block(h, gu.to_dev(d), None, empty, gu.to_dev(ctx), b4, p4)
    eb, ep = orc.pack_block_standard(d, ctx)
    np.testing.assert_array_equal(gu.to_np(b4), eb)
    np.testing.assert_array_equal(gu.to_np(p4), ep)
    t = np.array([1, 2], np.int32)
    rv.rv_pack_block_pending(h, gu.to_dev(t), gu.to_dev(d), None, empty, gu.to_dev(ctx), blk, pos)
    eb, ep = orc.pack_block_standard(np.concatenate([t[:, None], d], axis=1), ctx)
    np.testing.assert_array_equal(gu.to_np(blk), eb)
    np.testing.assert_array_equal(gu.to_np(pos), ep)
    with pytest.raises(rv.RVError):  # no template in standard verification
        rv.rv_pack_block(h, gu.to_dev(d), gu.to_dev(np.array([1], np.int32)), empty,
                         gu.to_dev(ctx), b4, p4)
    h.close()


# ------------------------------------------------------------------ full-size workloads

def test_llama3_8b_b1_full(gu):
    from paper_2505_18629_gb300 import synth
    _, _, gpu, ref, rep = _check(gu, synth.WORKLOADS["llama3-8b-b1"])
    assert rep.max_lse_err < 1e-3


def test_llama3_8b_b16_full(gu):
    from paper_2505_18629_gb300 import synth
    _check(gu, synth.WORKLOADS["llama3-8b-b16"])


def test_llama3_8b_b16_typical(gu):
    from paper_2505_18629_gb300 import rv, synth
    wl = synth.WORKLOADS["llama3-8b-b16"]
    inp = synth.generate(wl)
    drafts = gu.oracle_drafts(inp, ALPHA)
    eps, delta = _typical_params(gu, inp, drafts, ALPHA, "delta")
    h = gu.make_handle(wl)
    rv.rv_set_acceptance(h, rv.RV_ACCEPT_TYPICAL, eps, delta)
    gpu = gu.run_gpu(inp, drafts, ALPHA, h=h)
    ref = gu.oracle_typical(inp, drafts, ALPHA, eps, delta, with_attn=False)
    gu.compare(inp, drafts, ALPHA, ref, gpu, check_attn=False)
    h.close()


def test_llama3_70b_b32_sampled(gu):
    from paper_2505_18629_gb300 import synth
    _check(gu, synth.WORKLOADS["llama3-70b-b32"], seqs=[0, 17, 31])


# One sweep point per launch path (attention kernel, attention beside / before
# the LM head, LM-head kernel, sub-groups and chunks of its pairs, merge in
# the head's last CTA or a separate launch):
#   b1-g2-c1024   mma.sync attention beside the head; one-CTA head, merged in its last CTA
#   b4-g4-c8192   mma.sync attention before the head (KV capacity above 4608)
#   b4-g8-c1024   one-CTA head with 36 pairs (N = 80)
#   b16-g2-c1024  tcgen05 attention + chunk merge; CTA-pair head, 48 pairs, merged in its last CTA
#   b16-g4-c1024  CTA-pair head, 80 pairs, separate merge launch
#   b16-g4-c8192  as above with the attention before the head
#   b16-g8-c8192  CTA-pair head, 144 pairs in two sub-groups; attention before the head
#   b64-g2-c1024  CTA-pair head, two chunks of 96 pairs
#   b64-g4-c1024  CTA-pair head, two chunks of 160 pairs in two sub-groups
#   b64-g8-c8192  four chunks of 144 pairs in two sub-groups; attention before the head
@pytest.mark.parametrize("name", ["sweep-b1-g2-c1024", "sweep-b4-g4-c8192", "sweep-b4-g8-c1024",
                                  "sweep-b16-g2-c1024", "sweep-b16-g4-c1024",
                                  "sweep-b16-g4-c8192", "sweep-b16-g8-c8192",
                                  "sweep-b64-g2-c1024", "sweep-b64-g4-c1024",
                                  "sweep-b64-g8-c8192"])
def test_sweep_points(gu, name):
    from paper_2505_18629_gb300 import synth
    wl = synth.workload(name)
    seqs = None if wl.B <= 4 else ([0, 7, 15] if wl.B <= 16 else [0, 33, 63])
    _check(gu, wl, seqs=seqs)
