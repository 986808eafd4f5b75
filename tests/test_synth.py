"""Seeded input generator: determinism, shapes and the draft recipe."""
import numpy as np

from paper_2505_18629_gb300 import synth


def _small(**kw):
    base = synth.WORKLOADS["tiny"].replace(V=512, H=64, ctx=(3, 20), B=3)
    return base.replace(**kw)


def test_same_seed_same_inputs():
    a, b = synth.generate(_small()), synth.generate(_small())
    for f in ("W", "hidden", "q", "k_blk", "v_blk", "k_cache", "v_cache", "ctx_lens",
              "prompt_ids", "prefix_ids", "draft_keep", "draft_alt"):
        np.testing.assert_array_equal(getattr(a, f), getattr(b, f))
    c = synth.generate(_small(seed=5))
    assert not np.array_equal(a.W, c.W)


def test_shapes_and_ranges():
    wl = _small(dtype="bf16", gamma=5, R=8, Hq=8, Hkv=2, D=128)
    x = synth.generate(wl)
    assert wl.Lb == 18 and wl.Lh == 19
    assert x.W.shape == (512, 64) and x.W.dtype == np.uint16
    assert x.hidden.shape == (3, 19, 64)
    assert x.q.shape == (3, 18, 8, 128)
    assert x.k_cache.shape == (3, 2, 20 + 18, 128)
    assert x.prompt_ids.shape == (4,) and x.prefix_ids.shape == (3, 4)
    assert ((x.ctx_lens >= 3) & (x.ctx_lens <= 20)).all()
    assert ((x.draft_alt >= 0) & (x.draft_alt < 512)).all()


def test_hidden_rows_have_rms_one():
    wl = _small(dtype="bf16", hidden_rms1=True)
    h = synth.bf16_bits_to_f32(synth.generate(wl).hidden).astype(np.float64)
    np.testing.assert_allclose(np.sqrt((h ** 2).mean(-1)), 1.0, atol=1e-2)


def test_make_drafts_mixes_choice_and_alternative():
    x = synth.generate(_small(gamma=6, p_argmax=0.5))
    choice = np.full((3, 6), 7, np.int32)
    d = synth.make_drafts(x, choice)
    np.testing.assert_array_equal(d[x.draft_keep], 7)
    np.testing.assert_array_equal(d[~x.draft_keep], x.draft_alt[~x.draft_keep])


def test_zipf_alternatives_favour_low_ids():
    wl = _small(draft_dist="zipf1.1", gamma=8, B=64, V=4096)
    x = synth.generate(wl)
    assert np.median(x.draft_alt) < 4096 / 8


def test_bf16_round_trip():
    v = np.array([1.0, 0.1, -3.3, 1e-5], np.float32)
    back = synth.bf16_bits_to_f32(synth.to_bf16_bits(v))
    np.testing.assert_allclose(back, v, rtol=2 ** -8)
