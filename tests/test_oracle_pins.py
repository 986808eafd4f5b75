"""Pins of the CPU oracle against facts fixed outside the oracle itself.

Each test ties an oracle function to something it does not compute itself:
values the paper prints (Table 3 / Table 4 fixtures under tests/golden/),
closed forms, library routines (torch SDPA, scipy logsumexp / log_softmax),
invariants the paper states (Sec. 3.1 causality, Eq. 2 at alpha = 0 / 1), and
brute force on tiny inputs (lossless greedy exact-match verification).  The last
block plants plausible mistakes in the oracle and checks that a pin catches each.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import scipy.special
import torch

import oracle.rv_oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# --------------------------------------------------------------------------
# Block layout: Table 3 {5+3+4+5} and Alg. 1's m
# --------------------------------------------------------------------------

def test_table3_block_layout():
    g = _golden("table3_block_layout.json")
    gamma, n_prompt, n_prefix = g["gamma"], g["n_prompt"], g["n_prefix"]
    R = n_prompt + n_prefix
    drafts = np.array([[101, 102, 103, 104, 105]])
    prompt = np.array([201, 202, 203])
    prefix = np.array([[301, 302, 303, 304]])
    blk, pos = orc.pack_block(drafts, prompt, prefix, np.array([40]))
    assert blk.shape == (1, g["budget"])               # 5 + 3 + 4 + 5 = 17 inputs
    assert orc.m_index(gamma, R) == g["m"]
    b = blk[0]
    assert list(b[:gamma]) == list(drafts[0])
    assert list(b[gamma:gamma + n_prompt]) == list(prompt)
    assert list(b[gamma + n_prompt:gamma + R]) == list(prefix[0])
    assert list(b[gamma + R:]) == list(drafts[0])
    assert list(pos[0]) == list(range(40, 40 + g["budget"]))


@pytest.mark.parametrize("gamma,R", [(5, 7), (1, 0), (4, 4), (8, 8), (3, 1)])
def test_rows_score_their_draft(gamma, R):
    """Hidden row r predicts block token r; o_i and o_{m+i-1} must both score x_i.

    The original row of o_i predicts block position i-1 (first segment) and the
    reflective row predicts the copy's i-th token, for i = 1..gamma.
    """
    drafts = np.arange(1, gamma + 1)[None, :] + 1000
    prompt = np.arange(max(R - min(R, 4), 0)) + 2000
    prefix = (np.arange(min(R, 4)) + 3000)[None, :]
    blk, _ = orc.pack_block(drafts, prompt, prefix, np.array([0]))
    b = blk[0]
    Lb = b.shape[0]
    assert Lb == 2 * gamma + R
    for i in range(1, gamma + 1):
        assert b[orc.original_row(i)] == drafts[0, i - 1]
        assert b[orc.reflective_row(i, gamma, R)] == drafts[0, i - 1]
    # o_{gamma+1} / o_{m+gamma}: the rows after the last draft of each segment.
    assert orc.original_row(gamma + 1) == gamma
    assert orc.reflective_row(gamma + 1, gamma, R) == Lb


def test_table4_hyperparameters_are_the_defaults():
    from paper_2505_18629_gb300 import synth
    g = _golden("table4_hyperparameters.json")
    assert synth.DEFAULT_ALPHA == g["alpha"]
    assert synth.DEFAULT_PREFIX_LEN == g["prefix_len"]


# --------------------------------------------------------------------------
# Attention: torch SDPA (library), causality invariant, cache append
# --------------------------------------------------------------------------

def _rand_attn(rng, B, Lb, Hq, Hkv, D, ctx, cmax):
    q = rng.standard_normal((B, Lb, Hq, D))
    kb = rng.standard_normal((B, Lb, Hkv, D))
    vb = rng.standard_normal((B, Lb, Hkv, D))
    kc = rng.standard_normal((B, Hkv, cmax, D))
    vc = rng.standard_normal((B, Hkv, cmax, D))
    return q, kb, vb, kc, vc, np.asarray(ctx)


def _sdpa_reference(q, kb, vb, kc, vc, ctx):
    """torch.nn.functional.scaled_dot_product_attention, one sequence at a time."""
    B, Lb, Hq, D = q.shape
    Hkv = kb.shape[2]
    out = np.zeros_like(q)
    for b in range(B):
        c = int(ctx[b])
        K = np.concatenate([kc[b, :, :c], kb[b].transpose(1, 0, 2)], axis=1)   # [Hkv, c+Lb, D]
        Vv = np.concatenate([vc[b, :, :c], vb[b].transpose(1, 0, 2)], axis=1)
        Kt = torch.from_numpy(K).repeat_interleave(Hq // Hkv, dim=0)
        Vt = torch.from_numpy(Vv).repeat_interleave(Hq // Hkv, dim=0)
        Qt = torch.from_numpy(q[b].transpose(1, 0, 2).copy())                  # [Hq, Lb, D]
        mask = torch.ones(Lb, c + Lb, dtype=torch.bool)
        mask[:, c:] = torch.tril(torch.ones(Lb, Lb, dtype=torch.bool))
        o = torch.nn.functional.scaled_dot_product_attention(Qt, Kt, Vt, attn_mask=mask)
        out[b] = o.numpy().transpose(1, 0, 2)
    return out


@pytest.mark.parametrize("B,Lb,Hq,Hkv,D,ctx", [
    (1, 12, 4, 4, 16, [64]),          # tiny-config shape, MHA
    (2, 7, 8, 2, 16, [0, 5]),         # GQA, empty cache for one sequence
    (1, 1, 4, 1, 8, [9]),             # Lb = 1: plain decode attention
    (3, 5, 6, 3, 8, [3, 0, 11]),      # ragged contexts
])
def test_attention_matches_torch_sdpa(B, Lb, Hq, Hkv, D, ctx):
    rng = np.random.default_rng(7)
    args = _rand_attn(rng, B, Lb, Hq, Hkv, D, ctx, max(ctx) + Lb + 2)
    out, _, _ = orc.verify_attention(*args)
    ref = _sdpa_reference(*args)
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_attention_first_segment_unaffected_by_template_and_copy():
    """Sec. 3.1: the appended template and copy leave the first segment unchanged."""
    rng = np.random.default_rng(3)
    gamma, R = 4, 5
    Lb = 2 * gamma + R
    q, kb, vb, kc, vc, ctx = _rand_attn(rng, 2, Lb, 4, 2, 8, [6, 0], 30)
    full, _, _ = orc.verify_attention(q, kb, vb, kc, vc, ctx)
    first, _, _ = orc.verify_attention(q[:, :gamma], kb[:, :gamma], vb[:, :gamma], kc, vc, ctx)
    np.testing.assert_array_equal(full[:, :gamma], first)


def test_attention_appends_block_kv():
    rng = np.random.default_rng(4)
    q, kb, vb, kc, vc, ctx = _rand_attn(rng, 2, 3, 2, 2, 4, [2, 5], 10)
    _, kc2, vc2 = orc.verify_attention(q, kb, vb, kc, vc, ctx)
    for b, c in enumerate(ctx):
        np.testing.assert_array_equal(kc2[b, :, c:c + 3], kb[b].transpose(1, 0, 2))
        np.testing.assert_array_equal(vc2[b, :, c:c + 3], vb[b].transpose(1, 0, 2))
        np.testing.assert_array_equal(kc2[b, :, :c], kc[b, :, :c])
        np.testing.assert_array_equal(kc2[b, :, c + 3:], kc[b, :, c + 3:])


def test_widening_is_exact():
    x = np.array([1.0, -2.5, 3.140625, 65280.0, 1e-3], dtype=np.float32)
    bits = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    ref = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(orc.as_f64(bits), ref)


# --------------------------------------------------------------------------
# Head, log-softmax, fusion (Eq. 2)
# --------------------------------------------------------------------------

def test_logsumexp_closed_forms_and_library():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((5, 1000)) * 30
    np.testing.assert_allclose(orc.logsumexp(x), scipy.special.logsumexp(x, axis=-1), rtol=1e-13)
    c = 7.25
    assert orc.logsumexp(np.full((1, 4096), c))[0] == pytest.approx(c + math.log(4096), abs=1e-12)
    lp = x - orc.logsumexp(x)[:, None]
    np.testing.assert_allclose(np.exp(lp).sum(-1), 1.0, atol=1e-12)
    np.testing.assert_allclose(lp, scipy.special.log_softmax(x, axis=-1), atol=1e-12)


def _hand_example(alpha):
    """H=2, V=3: o = log[1,2,3] from hidden (1,0), o' = log[3,2,1] from (0,1)."""
    W = np.array([[0.0, math.log(3)], [math.log(2), math.log(2)], [math.log(3), 0.0]])
    gamma, R = 1, 1
    hidden = np.zeros((1, 2 * gamma + R + 1, 2))
    hidden[0, 0] = (1, 0)          # row of o_1
    hidden[0, 1] = (1, 0)          # row of o_2
    hidden[0, 2] = (0, 1)          # row of o_m     (reflective partner of o_1)
    hidden[0, 3] = (0, 1)          # row of o_{m+1}
    return orc.verify_head(W, hidden, np.array([[0]]), gamma, R, alpha)


def test_fusion_closed_form_alpha_03():
    """alpha = 0.3: p_1 is proportional to [3^0.3, 2, 3^0.7] (Eq. 2 by hand)."""
    r = _hand_example(0.3)
    w = np.array([3 ** 0.3, 2.0, 3 ** 0.7])
    assert r["lse_fused"][0, 0] == pytest.approx(math.log(w.sum()), abs=1e-14)
    assert r["logp_fused"][0, 0] == pytest.approx(math.log(w[0] / w.sum()), abs=1e-14)
    assert r["lse_orig"][0, 0] == pytest.approx(math.log(6), abs=1e-14)
    assert r["lse_refl"][0, 0] == pytest.approx(math.log(6), abs=1e-14)
    assert r["argmax"][0, 0] == 2
    assert r["margin"][0, 0] == pytest.approx(0.4 * math.log(3), abs=1e-14)   # z_2 - z_0


def test_fusion_closed_form_alpha_05_tie_breaks_low():
    """alpha = 0.5: p proportional to [sqrt3, 2, sqrt3]; argmax 1."""
    r = _hand_example(0.5)
    w = np.array([math.sqrt(3), 2.0, math.sqrt(3)])
    assert r["logp_fused"][0, 0] == pytest.approx(math.log(w[0] / w.sum()), abs=1e-14)
    assert r["argmax"][0, 0] == 1
    # alpha = 1 gives o' = log[3,2,1]: the argmax is token 0.
    assert _hand_example(1.0)["argmax"][0, 0] == 0


def _rand_head(rng, B, gamma, R, V, H):
    W = (rng.standard_normal((V, H)) * 0.5).astype(np.float32)
    hidden = rng.standard_normal((B, 2 * gamma + R + 1, H)).astype(np.float32)
    drafts = rng.integers(0, V, size=(B, gamma))
    return W, hidden, drafts


def _copy_rows(hidden, gamma, R):
    """Rows predicting the copy's tokens: block position Lb - gamma + i - 1 (i = 1..gamma+1)."""
    Lb = 2 * gamma + R
    return hidden[:, [Lb - gamma + i - 1 for i in range(1, gamma + 2)]]


@pytest.mark.parametrize("alpha", [0.0, 0.3, 1.0])
def test_fused_lse_is_lse_of_blended_hidden(alpha):
    """The head is linear (no bias): W((1-a)h_i + a h'_i) = (1-a) o_i + a o'_i."""
    rng = np.random.default_rng(11)
    gamma, R = 3, 5
    W, hidden, drafts = _rand_head(rng, 2, gamma, R, 300, 16)
    r = orc.verify_head(W, hidden, drafts, gamma, R, alpha)
    h_o = hidden[:, :gamma + 1].astype(np.float64)
    h_r = _copy_rows(hidden, gamma, R).astype(np.float64)
    blend = (1 - alpha) * h_o + alpha * h_r
    z = blend @ W.astype(np.float64).T
    np.testing.assert_allclose(r["lse_fused"], scipy.special.logsumexp(z, axis=-1), atol=1e-10)
    np.testing.assert_allclose(r["lse_orig"],
                               scipy.special.logsumexp(h_o @ W.astype(np.float64).T, axis=-1),
                               atol=1e-10)
    np.testing.assert_allclose(r["lse_refl"],
                               scipy.special.logsumexp(h_r @ W.astype(np.float64).T, axis=-1),
                               atol=1e-10)
    lsm = scipy.special.log_softmax(z, axis=-1)
    bi, ii = np.arange(2)[:, None], np.arange(gamma)[None, :]
    np.testing.assert_allclose(r["logp_fused"], lsm[bi, ii, drafts], atol=1e-10)


def test_alpha_zero_is_standard_verification():
    """Eq. 2 at alpha = 0: p_i = softmax(o_i), the standard target distribution."""
    rng = np.random.default_rng(12)
    gamma, R = 4, 4
    W, hidden, drafts = _rand_head(rng, 3, gamma, R, 200, 8)
    r = orc.verify_head(W, hidden, drafts, gamma, R, 0.0)
    np.testing.assert_array_equal(r["lse_fused"], r["lse_orig"])
    np.testing.assert_array_equal(r["logp_fused"], r["logp_orig"])
    o = hidden[:, :gamma + 1].astype(np.float64) @ W.astype(np.float64).T
    np.testing.assert_array_equal(r["argmax"], np.argmax(o, axis=-1))


def test_margin_from_sorted_logits():
    rng = np.random.default_rng(13)
    gamma, R = 3, 2
    W, hidden, drafts = _rand_head(rng, 4, gamma, R, 50, 6)
    drafts[0, 0] = 0
    r = orc.verify_head(W, hidden, drafts, gamma, R, 0.3)
    z = r["z"]
    for b in range(4):
        for i in range(gamma):
            s = np.sort(z[b, i])
            zx = z[b, i, drafts[b, i]]
            want = s[-1] - s[-2] if zx == s[-1] else s[-1] - zx
            assert r["margin"][b, i] == pytest.approx(want, abs=1e-12)
        for i in range(gamma + 1):
            s = np.sort(z[b, i])
            assert r["choice_gap"][b, i] == pytest.approx(s[-1] - s[-2], abs=1e-12)
            assert z[b, i, r["argmax"][b, i]] == s[-1]


# --------------------------------------------------------------------------
# Acceptance (Alg. 2, greedy): lossless w.r.t. greedy decoding, brute force
# --------------------------------------------------------------------------

def _greedy_tables(rng, gamma, V):
    """Random distinct-valued per-position greedy choices x^_1..x^_{gamma+1}."""
    z = rng.standard_normal((1, gamma + 1, V))
    return orc.greedy_choice(z)[0]


@pytest.mark.parametrize("V,gamma", [(3, 1), (4, 2), (5, 3), (6, 3)])
def test_accept_is_lossless_greedy_decoding_brute_force(V, gamma):
    """Every draft tuple in V^gamma: the output [x_1..x_n, t] is exactly the
    first n+1 tokens of greedy decoding, and n is maximal (x_{n+1} differs)."""
    rng = np.random.default_rng(V * 10 + gamma)
    for _ in range(3):
        g = _greedy_tables(rng, gamma, V)
        for d in itertools.product(range(V), repeat=gamma):
            d = np.array(d)[None, :]
            acc, n, t = orc.exact_match_accept(d, g[None, :])
            n, t = int(n[0]), int(t[0])
            out = list(d[0, :n]) + [t]
            assert out == list(g[:n + 1])
            assert 0 <= n <= gamma
            assert (n == gamma) == bool(acc.all())
            if n < gamma:
                assert d[0, n] != g[n]
            assert acc[0, :n].all()


def test_literal_alg2_set_is_not_lossless():
    """The stopping set as printed (first MATCH) breaks losslessness; the
    first-mismatch reading used by the oracle keeps it."""
    g = np.array([[1, 2, 0]])
    d = np.array([[0, 2]])          # x_1 rejected, x_2 happens to match
    literal_n = min([i - 1 for i in range(1, 3) if d[0, i - 1] == g[0, i - 1]] + [2])
    literal_out = list(d[0, :literal_n]) + [g[0, literal_n]]
    assert literal_out == [0, 2] and literal_out != list(g[0, :literal_n + 1])
    _, n, t = orc.exact_match_accept(d, g)
    assert int(n[0]) == 0 and int(t[0]) == 1


def test_verify_step_end_to_end_small():
    rng = np.random.default_rng(21)
    B, gamma, R, V, H = 2, 3, 4, 64, 8
    Lb = 2 * gamma + R
    W = rng.standard_normal((V, H)).astype(np.float32)
    hidden = rng.standard_normal((B, Lb + 1, H)).astype(np.float32)
    q, kb, vb, kc, vc, ctx = _rand_attn(rng, B, Lb, 2, 1, 4, [3, 9], 30)
    first = orc.verify_head(W, hidden, np.zeros((B, gamma), np.int64), gamma, R, 0.3)["argmax"]
    drafts = first[:, :gamma].copy()
    drafts[1, 1] = (drafts[1, 1] + 1) % V              # sequence 1 rejects x_2
    r = orc.verify_step(W, hidden, q, kb, vb, kc, vc, ctx, drafts, np.array([5, 6]),
                        np.array([[1, 2], [3, 4]]), gamma, R, 0.3)
    assert list(r["accepted_len"]) == [3, 1]
    assert list(r["ctx_out"]) == [6, 10]
    assert r["next_token"][0] == r["argmax"][0, 3]
    assert r["next_token"][1] == r["argmax"][1, 1]


# --------------------------------------------------------------------------
# Planted mistakes: each plausible slip in the oracle must fail a pin above
# --------------------------------------------------------------------------

def _fails(fn):
    try:
        fn()
    except AssertionError:
        return True
    return False


def test_pins_catch_off_by_one_shift(monkeypatch):
    monkeypatch.setattr(orc, "shift_len", lambda gamma, R: gamma + R - 1)
    assert _fails(lambda: test_rows_score_their_draft(5, 7))
    assert _fails(lambda: test_fused_lse_is_lse_of_blended_hidden(0.3))


def test_pins_catch_swapped_alpha(monkeypatch):
    monkeypatch.setattr(orc, "fuse", lambda o, r, a: a * o + (1 - a) * r)
    assert _fails(test_fusion_closed_form_alpha_03)
    assert _fails(lambda: test_fused_lse_is_lse_of_blended_hidden(0.3))


def test_pins_catch_literal_stopping_rule(monkeypatch):
    def literal(drafts, choice):
        drafts, choice = np.asarray(drafts), np.asarray(choice)
        B, gamma = drafts.shape
        acc = drafts == choice[:, :gamma]
        n = np.array([min([i - 1 for i in range(1, gamma + 1) if acc[b, i - 1]] + [gamma])
                      for b in range(B)])
        return acc.astype(np.uint8), n, choice[np.arange(B), n]
    monkeypatch.setattr(orc, "exact_match_accept", literal)
    assert _fails(lambda: test_accept_is_lossless_greedy_decoding_brute_force(4, 2))


def test_pins_catch_dropped_causal_mask(monkeypatch):
    real = orc.verify_attention

    def no_mask(q, k_blk, v_blk, k_cache, v_cache, ctx_lens):
        # planted slip: every block query sees the whole block
        out, kc, vc = real(q, k_blk, v_blk, k_cache, v_cache, ctx_lens)
        qf, kb, vb = orc.as_f64(q), orc.as_f64(k_blk), orc.as_f64(v_blk)
        B, Lb, Hq, D = qf.shape
        G = Hq // kb.shape[2]
        for b in range(B):
            c = int(ctx_lens[b])
            for h in range(Hq):
                keys = np.concatenate([orc.as_f64(k_cache)[b, h // G, :c], kb[b, :, h // G]])
                vals = np.concatenate([orc.as_f64(v_cache)[b, h // G, :c], vb[b, :, h // G]])
                for j in range(Lb):
                    s = keys @ qf[b, j, h] / np.sqrt(D)
                    w = np.exp(s - s.max())
                    out[b, j, h] = (w / w.sum()) @ vals
        return out, kc, vc
    monkeypatch.setattr(orc, "verify_attention", no_mask)
    assert _fails(lambda: test_attention_matches_torch_sdpa(2, 7, 8, 2, 16, [0, 5]))
    assert _fails(test_attention_first_segment_unaffected_by_template_and_copy)


# ------------------------------------------------------------------ Alg. 3: typical acceptance

def test_entropy_closed_forms_and_library():
    import scipy.stats
    rng = np.random.default_rng(11)
    # constant logits: the uniform distribution, H = ln V
    for V in (2, 3, 1000):
        assert abs(orc.entropy(np.full(V, 3.7)) - math.log(V)) < 1e-12
    # two outcomes with logits (0, a): the binary entropy of sigma(a)
    for a in (-3.0, 0.0, 0.5, 7.0):
        p = 1.0 / (1.0 + math.exp(-a))
        h = -(p * math.log(p) + (1 - p) * math.log(1 - p))
        assert abs(orc.entropy(np.array([0.0, a])) - h) < 1e-12
    # a library routine on random logits, batched along an axis
    x = rng.normal(0, 3, (4, 5, 257))
    ref = scipy.stats.entropy(scipy.special.softmax(x, axis=-1), axis=-1)
    np.testing.assert_allclose(orc.entropy(x), ref, rtol=1e-12, atol=1e-12)
    # a nearly one-hot distribution has (almost) no entropy; bounds 0 <= H <= ln V
    assert 0.0 <= orc.entropy(np.array([200.0, 0.0, 0.0])) < 1e-80
    h = orc.entropy(x)
    assert (h >= 0).all() and (h <= math.log(257) + 1e-12).all()


def test_entropy_in_head_is_of_the_unfused_original_logits():
    # H(p_original) does not depend on alpha; at alpha = 0 the fused
    # distribution is the original one, so it equals the fused entropy there
    rng = np.random.default_rng(12)
    V, H, gamma, R = 50, 8, 3, 2
    W = rng.normal(0, 1, (V, H))
    hidden = rng.normal(0, 1, (2, 2 * gamma + R + 1, H))
    drafts = rng.integers(0, V, (2, gamma))
    a0 = orc.verify_head(W, hidden, drafts, gamma, R, 0.0)
    a1 = orc.verify_head(W, hidden, drafts, gamma, R, 0.7)
    np.testing.assert_array_equal(a0["ent_orig"], a1["ent_orig"])
    np.testing.assert_allclose(a0["ent_orig"], orc.entropy(a0["z"]), atol=1e-12)
    assert not np.allclose(a1["ent_orig"], orc.entropy(a1["z"]))


def test_typical_threshold_worked_example():
    # uniform original distribution over V = 3: H = ln 3, so with delta = 0.3
    # the entropy term is 0.3 / 3 = 0.1 and eps = 0.09 is the binding side
    H = np.full((1, 3), math.log(3))
    logp = np.log(np.array([[0.5, 0.2, 0.05]]))  # kept, kept, rejected
    choice = np.array([[4, 5, 6]])
    acc, n, t, gap = orc.typical_accept(np.zeros((1, 2)), logp[:, :2], H, choice, 0.09, 0.3)
    assert acc.tolist() == [[True, True]] and n[0] == 2 and t[0] == 6
    acc, n, t, gap = orc.typical_accept(np.zeros((1, 3)), logp, H, np.array([[4, 5, 6, 7]]), 0.09, 0.3)
    assert acc.tolist() == [[True, True, False]] and n[0] == 2 and t[0] == 6
    np.testing.assert_allclose(gap[0], np.log([0.5, 0.2, 0.05]) - math.log(0.09), atol=1e-12)
    # a low-entropy original distribution lowers the threshold to delta * e^-H
    acc, n, t, gap = orc.typical_accept(np.zeros((1, 1)), np.log([[0.05]]), np.array([[3.0]]),
                                        np.array([[1, 2]]), 0.09, 0.3)
    assert acc[0, 0] and abs(gap[0, 0] - (math.log(0.05) - (math.log(0.3) - 3.0))) < 1e-12


def test_typical_accept_sampled_t_law_and_greedy_limit():
    # Alg. 3 with t ~ p_{n+1} at temperature T: over a fine grid of uniforms
    # the frequency of each t is softmax(z_{n+1} / T) (the inverse CDF's law);
    # the kept drafts and n are typical_accept's; T -> 0 gives its greedy t
    B, gamma, V = 2, 3, 5
    z = np.array([[[0.0, 1.0, 2.0, 0.5, -1.0]] * (gamma + 1),
                  [[3.0, 0.0, 0.0, 2.9, 1.0]] * (gamma + 1)])
    logp = np.log(np.array([[0.5, 0.01, 0.4], [0.3, 0.3, 0.3]]))
    H = np.full((B, gamma + 1), 1.0)
    acc_g, n_g, t_g, _ = orc.typical_accept(np.zeros((B, gamma)), logp, H,
                                            z.argmax(axis=-1), 0.2, 0.3)
    for T in (1.0, 0.5):
        K = 20000
        counts = np.zeros((B, V))
        for k in range(K):
            u = np.full((B, gamma + 1), (k + 0.5) / K)
            acc, n, t, _, _ = orc.typical_accept_sampled(np.zeros((B, gamma)), logp, H, z, 0.2, 0.3,
                                                         T, u)
            assert (acc == acc_g).all() and (n == n_g).all()
            counts[np.arange(B), t] += 1
        for b in range(B):
            zt = z[b, n_g[b]] / T
            p = np.exp(zt - zt.max())
            p /= p.sum()
            np.testing.assert_allclose(counts[b] / K, p, atol=2.0 / K)
    u = np.full((B, gamma + 1), 0.37)
    _, _, t0, _, _ = orc.typical_accept_sampled(np.zeros((B, gamma)), logp, H, z, 0.2, 0.3, 1e-6, u)
    assert (t0 == t_g).all()


def test_typical_accept_limits_and_monotonicity():
    rng = np.random.default_rng(13)
    B, gamma = 64, 6
    logp = np.log(rng.uniform(1e-4, 1.0, (B, gamma)))
    H = rng.uniform(0.0, 6.0, (B, gamma + 1))
    choice = rng.integers(0, 1000, (B, gamma + 1))
    # threshold above every probability: nothing is kept, t = the first choice
    acc, n, t, _ = orc.typical_accept(np.zeros((B, gamma)), logp, H, choice, 2.0, 1e9)
    assert not acc.any() and (n == 0).all() and (t == choice[:, 0]).all()
    # a vanishing threshold keeps every draft, t = the bonus position's choice
    acc, n, t, _ = orc.typical_accept(np.zeros((B, gamma)), logp, H, choice, 1e-300, 1e-300)
    assert acc.all() and (n == gamma).all() and (t == choice[:, gamma]).all()
    # n is the number of leading kept drafts, and falls as eps or delta grow
    prev = None
    for eps in (1e-3, 1e-2, 0.05, 0.1, 0.3):
        acc, n, t, _ = orc.typical_accept(np.zeros((B, gamma)), logp, H, choice, eps, 0.3)
        for b in range(B):
            assert acc[b, :n[b]].all() and (n[b] == gamma or not acc[b, n[b]])
            assert t[b] == choice[b, n[b]]
        if prev is not None:
            assert (n <= prev).all()
        prev = n


def test_pins_catch_fused_entropy(monkeypatch):
    real = orc.verify_head

    def fused_entropy(W, hidden, drafts, gamma, R, alpha):
        out = real(W, hidden, drafts, gamma, R, alpha)
        out["ent_orig"] = orc.entropy(out["z"])  # planted slip: entropy of p_i, not p_original
        return out
    monkeypatch.setattr(orc, "verify_head", fused_entropy)
    assert _fails(test_entropy_in_head_is_of_the_unfused_original_logits)


def test_pins_catch_swapped_threshold_parameters(monkeypatch):
    def swapped(drafts, logp_fused, ent_orig, choice, eps, delta):
        # planted slip: eps and delta exchanged in the threshold
        return real(drafts, logp_fused, ent_orig, choice, delta, eps)
    real = orc.typical_accept
    monkeypatch.setattr(orc, "typical_accept", swapped)
    assert _fails(test_typical_threshold_worked_example)


# ------------------------------------------------------------------ Alg. 1: speculative sampling

def test_inverse_cdf_sample_closed_forms():
    w = np.array([0.1, 0.0, 0.3, 0.6])
    assert orc.inverse_cdf_sample(w, 0.0) == 0
    assert orc.inverse_cdf_sample(w, 0.0999) == 0
    assert orc.inverse_cdf_sample(w, 0.1001) == 2          # a zero weight is never drawn
    assert orc.inverse_cdf_sample(w, 0.3999) == 2
    assert orc.inverse_cdf_sample(w, 0.4001) == 3
    assert orc.inverse_cdf_sample(w, 0.999999) == 3
    assert orc.inverse_cdf_sample(5.0 * w, 0.25) == 2       # scale-free
    # weights ending in zeros: the top of the range takes the last weighted token
    tail0 = np.array([0.5, 0.5, 0.0])
    assert orc.inverse_cdf_sample(tail0, np.nextafter(1.0, 0.0)) == 1
    assert orc.inverse_cdf_sample(tail0, 1.0) == 1
    # a midpoint grid of u reproduces w / sum(w) exactly
    grid = (np.arange(1000) + 0.5) / 1000
    hits = np.bincount([orc.inverse_cdf_sample(w, x) for x in grid], minlength=4) / 1000
    np.testing.assert_allclose(hits, w / w.sum(), atol=1e-3)


def _spec_case(rng, B, gamma, V, same=False):
    z = rng.normal(0, 1.5, (B, gamma + 1, V))
    q = scipy.special.softmax(rng.normal(0, 1.5, (B, gamma, V)), axis=-1)
    if same:
        q = scipy.special.softmax(z[:, :gamma], axis=-1)
    drafts = np.array([[rng.choice(V, p=q[b, i]) for i in range(gamma)] for b in range(B)])
    return z, q, drafts


def test_speculative_draft_equal_to_target_accepts_everything():
    # q_i = p_i: every ratio is 1 and r_i < 1 keeps every draft; t ~ p_{gamma+1}
    rng = np.random.default_rng(21)
    z, q, drafts = _spec_case(rng, 8, 4, 11, same=True)
    r = rng.uniform(0, 1, (8, 4))
    u = rng.uniform(0, 1, 8)
    acc, n, t, lr, _ = orc.speculative_accept(drafts, z, q, r, u)
    assert acc.all() and (n == 4).all()
    np.testing.assert_allclose(lr, 0.0, atol=1e-12)
    p_last = scipy.special.softmax(z[:, 4], axis=-1)
    for b in range(8):
        assert t[b] == orc.inverse_cdf_sample(p_last[b], u[b])


def test_speculative_first_token_is_distributed_as_p1():
    # The speculative-sampling guarantee (Alg. 1): over x_1 ~ q_1, r_1 and u the
    # first emitted token (x_1 if kept, else t) has distribution p_1 exactly.
    # Evaluated by quadrature with the oracle itself: a midpoint grid of r_1
    # gives P(keep x_1), and a midpoint grid of u the law of t after a rejection.
    rng = np.random.default_rng(22)
    V, gamma = 6, 1
    z = rng.normal(0, 1.0, (1, gamma + 1, V))
    q = scipy.special.softmax(rng.normal(0, 1.0, (1, gamma, V)), axis=-1)
    p1 = scipy.special.softmax(z[0, 0])
    r_grid = (np.arange(2000) + 0.5) / 2000
    u_grid = (np.arange(2000) + 0.5) / 2000
    dist = np.zeros(V)
    for x1 in range(V):
        d = np.array([[x1]])
        keep = np.mean([orc.speculative_accept(d, z, q, np.array([[r1]]), np.array([0.5]))[0][0, 0]
                        for r1 in r_grid])
        dist[x1] += q[0, 0, x1] * keep
        if keep < 1.0:
            for uu in u_grid:  # r_1 just below 1 rejects every draft with p_1(x_1) < q_1(x_1)
                t = orc.speculative_accept(d, z, q, np.array([[1 - 1e-12]]), np.array([uu]))[2][0]
                dist[t] += q[0, 0, x1] * (1.0 - keep) / len(u_grid)
    np.testing.assert_allclose(dist, p1, atol=2e-3)
    assert abs(dist.sum() - 1.0) < 1e-9


def test_speculative_stopping_and_residual():
    rng = np.random.default_rng(23)
    B, gamma, V = 32, 5, 9
    z, q, drafts = _spec_case(rng, B, gamma, V)
    r = rng.uniform(0, 1, (B, gamma))
    u = rng.uniform(0, 1, B)
    acc, n, t, lr, gap = orc.speculative_accept(drafts, z, q, r, u)
    p = scipy.special.softmax(z, axis=-1)
    for b in range(B):
        assert acc[b, :n[b]].all() and (n[b] == gamma or not acc[b, n[b]])
        if n[b] < gamma:
            w = np.maximum(0, p[b, n[b]] - q[b, n[b]])
            assert w[t[b]] > 0                                 # t lies where p exceeds q
            # the residual never proposes the rejected draft more than p allows
        else:
            assert p[b, gamma, t[b]] > 0
    # r = 0 keeps every draft with p_i(x_i) > 0; r -> 1 keeps only drafts with p >= q
    acc0, n0, *_ = orc.speculative_accept(drafts, z, q, np.full((B, gamma), 1e-300), u)
    assert acc0.all() and (n0 == gamma).all()
    acc1, *_ = orc.speculative_accept(drafts, z, q, np.full((B, gamma), 1 - 1e-12), u)
    np.testing.assert_array_equal(acc1, lr >= np.log1p(-1e-12))


def test_pins_catch_plain_p_instead_of_residual(monkeypatch):
    real = orc.speculative_accept

    def plain(drafts, z, q, r, u):
        # planted slip: t ~ p_{n+1} even after a rejection (no residual)
        acc, n, t, lr, gap = real(drafts, z, q, r, u)
        logp = np.asarray(z) - orc.logsumexp(np.asarray(z))[..., None]
        t = np.array([orc.inverse_cdf_sample(np.exp(logp[b, n[b]]), float(u[b]))
                      for b in range(len(n))])
        return acc, n, t, lr, gap
    monkeypatch.setattr(orc, "speculative_accept", plain)
    assert _fails(test_speculative_first_token_is_distributed_as_p1)


# ------------------------------------------------------------------ Alg. 2: sampled exact match

def test_sampled_exact_low_temperature_is_greedy():
    # T -> 0: softmax(z / T) concentrates on argmax z, so every draw is the
    # greedy choice whatever u is, and the rule is the greedy exact match.
    rng = np.random.default_rng(31)
    B, gamma, V = 16, 5, 13
    z = rng.normal(0, 2.0, (B, gamma + 1, V))
    greedy = orc.greedy_choice(z)
    drafts = np.where(rng.uniform(size=(B, gamma)) < 0.7, greedy[:, :gamma],
                      rng.integers(0, V, (B, gamma)))
    u = rng.uniform(0, 1, (B, gamma + 1))
    acc, n, t, xhat, _ = orc.sampled_exact_accept(drafts, z, 1e-4, u)
    np.testing.assert_array_equal(xhat, greedy)
    acc_g, n_g, t_g = orc.exact_match_accept(drafts, greedy)
    np.testing.assert_array_equal(acc, acc_g)
    np.testing.assert_array_equal(n, n_g)
    np.testing.assert_array_equal(t, t_g)


@pytest.mark.parametrize("T", [0.2, 0.8, 1.0, 3.0])
def test_sampled_exact_temperature_closed_form(T):
    # Two tokens with logits (0, d): P(x^ = 1) = 1 / (1 + exp(-d / T)).  A
    # midpoint grid of u gives the draw frequencies to within 1 / grid.
    d = 0.9
    z = np.array([[[0.0, d]]])
    grid = (np.arange(4000) + 0.5) / 4000
    ones = np.mean([orc.sampled_exact_accept(np.zeros((1, 0), np.int64), z, T,
                                             np.array([[x]]))[3][0, 0] for x in grid])
    assert abs(ones - 1.0 / (1.0 + np.exp(-d / T))) < 1e-3


def test_sampled_exact_emits_the_target_draws():
    # Lossless: the emitted tokens [x_1..x_n, t] are the target's own draws
    # x^_1..x^_{n+1}, so the output is what sampling the target alone gives.
    rng = np.random.default_rng(32)
    B, gamma, V = 64, 6, 7
    z = rng.normal(0, 1.0, (B, gamma + 1, V))
    T = 0.8
    u = rng.uniform(0, 1, (B, gamma + 1))
    p_t = scipy.special.softmax(z / T, axis=-1)
    # drafts that often agree with the draws: x_i ~ p_t (an ideal draft model)
    drafts = np.array([[rng.choice(V, p=p_t[b, i]) for i in range(gamma)] for b in range(B)])
    acc, n, t, xhat, _ = orc.sampled_exact_accept(drafts, z, T, u)
    assert (n > 0).any() and (n < gamma).any()
    for b in range(B):
        emitted = list(drafts[b, :n[b]]) + [t[b]]
        assert emitted == list(xhat[b, :n[b] + 1])
        assert n[b] == gamma or drafts[b, n[b]] != xhat[b, n[b]]
        for i in range(gamma + 1):
            assert xhat[b, i] == orc.inverse_cdf_sample(p_t[b, i], u[b, i])


def test_pins_catch_sampled_exact_fresh_draw_for_t(monkeypatch):
    real = orc.sampled_exact_accept

    def fresh(drafts, z, temperature, u):
        # planted slip: t drawn afresh from p_{n+1} instead of reusing x^_{n+1}
        acc, n, t, xhat, gap = real(drafts, z, temperature, u)
        zt = np.asarray(z, np.float64) / temperature
        p_t = np.exp(zt - orc.logsumexp(zt)[..., None])
        t = np.array([orc.inverse_cdf_sample(p_t[b, n[b]], 1.0 - float(u[b, n[b]]))
                      for b in range(len(n))])
        return acc, n, t, xhat, gap
    monkeypatch.setattr(orc, "sampled_exact_accept", fresh)
    assert _fails(test_sampled_exact_emits_the_target_draws)


def test_pins_catch_temperature_multiplied(monkeypatch):
    real = orc.sampled_exact_accept
    # planted slip: softmax(z * T) instead of softmax(z / T)
    monkeypatch.setattr(orc, "sampled_exact_accept",
                        lambda drafts, z, T, u: real(drafts, np.asarray(z) * T * T, T, u))
    assert _fails(lambda: test_sampled_exact_temperature_closed_form(0.2))


# --------------------------------------------------------------------------
# Pending-token block [t, x_1..x_gamma, template, x_1..x_gamma]
# --------------------------------------------------------------------------

def test_pending_block_layout_table3():
    # Table 3's {5+3+4+5} block with the last emitted token in front: 18 positions
    g = _golden("table3_block_layout.json")
    gamma, n_prompt, n_prefix = g["gamma"], g["n_prompt"], g["n_prefix"]
    drafts = np.array([[101, 102, 103, 104, 105], [111, 112, 113, 114, 115]])
    prompt = np.array([201, 202, 203])
    prefix = np.array([[301, 302, 303, 304], [311, 312, 313, 314]])
    ctx = np.array([40, 7])
    blk, pos = orc.pack_block_pending(np.array([99, 98]), drafts, prompt, prefix, ctx)
    std, _ = orc.pack_block(drafts, prompt, prefix, ctx)
    assert blk.shape == (2, g["budget"] + 1)
    assert list(blk[:, 0]) == [99, 98]
    np.testing.assert_array_equal(blk[:, 1:], std)
    for b in range(2):
        assert list(pos[b]) == list(range(ctx[b], ctx[b] + g["budget"] + 1))


@pytest.mark.parametrize("gamma,R", [(5, 7), (1, 0), (4, 4)])
def test_pending_rows_score_their_draft(gamma, R):
    # hidden row r follows pending-block position r and predicts position r + 1:
    # row 0 (the pending token) predicts x_1, and the head's original /
    # reflective rows (unchanged from the standard layout) score x_i twice
    drafts = np.arange(1, gamma + 1)[None, :] + 1000
    prompt = np.arange(max(R - min(R, 4), 0)) + 2000
    prefix = (np.arange(min(R, 4)) + 3000)[None, :]
    blk, _ = orc.pack_block_pending(np.array([7]), drafts, prompt, prefix, np.array([0]))
    b = blk[0]
    for i in range(1, gamma + 1):
        assert b[orc.original_row(i) + 1] == drafts[0, i - 1]
        assert b[orc.reflective_row(i, gamma, R) + 1] == drafts[0, i - 1]
    assert orc.reflective_row(gamma + 1, gamma, R) == b.shape[0] - 1   # the last position


def _pending_attention_case(rng, B=3, gamma=3, R=2, Hq=4, Hkv=2, D=8, ctxs=(0, 5, 11)):
    Lp = 2 * gamma + R + 1
    C = max(ctxs) + Lp + 2
    q = rng.normal(size=(B, Lp, Hq, D))
    kb = rng.normal(size=(B, Lp, Hkv, D))
    vb = rng.normal(size=(B, Lp, Hkv, D))
    kc = rng.normal(size=(B, Hkv, C, D))
    vc = rng.normal(size=(B, Hkv, C, D))
    return q, kb, vb, kc, vc, np.asarray(ctxs)


def test_pending_attention_equals_standard_after_appending_t():
    # Causality (Sec. 3.1): running the pending block at ctx is the same forward
    # pass as first appending t's key/value at position ctx and running the
    # standard block at ctx + 1 -- same outputs for the block's other rows, same
    # cache afterwards; and t's own row is plain decoding over context + t.
    rng = np.random.default_rng(31)
    q, kb, vb, kc, vc, ctx = _pending_attention_case(rng)
    out, kc1, vc1 = orc.verify_attention(q, kb, vb, kc, vc, ctx)
    kc2, vc2 = kc.copy(), vc.copy()
    for b in range(len(ctx)):
        kc2[b, :, ctx[b]] = kb[b, 0]
        vc2[b, :, ctx[b]] = vb[b, 0]
    out2, kc3, vc3 = orc.verify_attention(q[:, 1:], kb[:, 1:], vb[:, 1:], kc2, vc2, ctx + 1)
    np.testing.assert_allclose(out[:, 1:], out2, rtol=0, atol=1e-12)
    np.testing.assert_array_equal(kc1, kc3)
    np.testing.assert_array_equal(vc1, vc3)
    dec, _, _ = orc.verify_attention(q[:, :1], kb[:, :1], vb[:, :1], kc, vc, ctx)
    np.testing.assert_allclose(out[:, :1], dec, rtol=0, atol=1e-12)


def test_pending_step_keeps_t_and_the_accepted_drafts():
    # After the step the context is [old context, t, x_1..x_n]: its last kept
    # key is x_n's (t's when n = 0) and t's key sits at the old length.
    from paper_2505_18629_gb300 import synth
    wl = synth.Workload("p", B=4, gamma=3, R=2, ctx=(0, 20), H=32, Hq=4, Hkv=2, D=16, V=50,
                        dtype="f32", p_argmax=0.5, seed=33)
    inp = synth.generate(wl)
    Lp = wl.Lb + 1
    rng = np.random.default_rng(34)
    q = rng.normal(size=(wl.B, Lp, wl.Hq, wl.D)).astype(np.float32)
    kb = rng.normal(size=(wl.B, Lp, wl.Hkv, wl.D)).astype(np.float32)
    vb = rng.normal(size=(wl.B, Lp, wl.Hkv, wl.D)).astype(np.float32)
    kc = np.zeros((wl.B, wl.Hkv, wl.capacity + 1, wl.D), np.float32)
    vc = np.zeros_like(kc)
    choice = orc.verify_head(inp.W, inp.hidden, np.zeros((wl.B, wl.gamma), np.int64), wl.gamma,
                             wl.R, 0.3)["argmax"]
    drafts = np.where(rng.uniform(size=(wl.B, wl.gamma)) < 0.6, choice[:, :wl.gamma],
                      rng.integers(0, wl.V, (wl.B, wl.gamma)))
    pending = rng.integers(0, wl.V, wl.B)
    r = orc.verify_step_pending(inp.W, inp.hidden, q, kb, vb, kc, vc, inp.ctx_lens, pending,
                                drafts, inp.prompt_ids, inp.prefix_ids, wl.gamma, wl.R, 0.3)
    assert (r["block_ids"][:, 0] == pending).all()
    for b in range(wl.B):
        c, n, co = int(inp.ctx_lens[b]), int(r["accepted_len"][b]), int(r["ctx_out"][b])
        np.testing.assert_array_equal(r["k_cache"][b, :, c], kb[b, 0])          # t
        np.testing.assert_array_equal(r["k_cache"][b, :, co - 1], kb[b, n])     # x_n (or t)
        assert co - c - 1 == n
    # the emitted tokens are those of the standard layout's step (same head rows)
    std = orc.exact_match_accept(drafts, r["argmax"])
    np.testing.assert_array_equal(r["accepted_len"], std[1])
    np.testing.assert_array_equal(r["next_token"], std[2])


def test_pins_catch_pending_length_without_t(monkeypatch):
    real = orc.verify_step_pending

    def drop_t(*args, **kw):
        r = real(*args, **kw)
        r["ctx_out"] = r["ctx_out"] - 1
        return r
    monkeypatch.setattr(orc, "verify_step_pending", drop_t)
    with pytest.raises(AssertionError):
        test_pending_step_keeps_t_and_the_accepted_drafts()


def test_pins_catch_pending_token_at_the_end(monkeypatch):
    real = orc.pack_block

    def t_last(pending, drafts, prompt_ids, prefix_ids, ctx_lens):
        blk, pos = real(drafts, prompt_ids, prefix_ids, ctx_lens)
        blk = np.concatenate([blk, np.asarray(pending)[:, None]], axis=1).astype(np.int32)
        pos = (np.asarray(ctx_lens)[:, None] + np.arange(blk.shape[1])).astype(np.int32)
        return blk, pos
    monkeypatch.setattr(orc, "pack_block_pending", t_last)
    with pytest.raises(AssertionError):
        test_pending_block_layout_table3()


# --------------------------------------------------------------------------
# Pre-blended head: z_i = W b_i, b_i the bf16-rounded blend (linearity of Eq. 2)
# --------------------------------------------------------------------------

def test_round_to_bf16_matches_torch():
    rng = np.random.default_rng(41)
    x = np.concatenate([rng.normal(0, 1, 20000), rng.normal(0, 1e-30, 100), rng.normal(0, 1e30, 100),
                        [1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -(1.0 + 2 ** -8), 0.0, -0.0, 2 ** -130]])
    x = x.astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(orc.round_to_bf16(x), ref)


def _preblend_case(seed, B=3, gamma=3, R=2, H=48, V=40):
    from paper_2505_18629_gb300 import synth
    rng = np.random.default_rng(seed)
    W = synth.to_bf16_bits(rng.normal(0, 0.05, (V, H)).astype(np.float32))
    hidden = synth.to_bf16_bits(rng.normal(0, 1, (B, 2 * gamma + R + 1, H)).astype(np.float32))
    drafts = rng.integers(0, V, (B, gamma))
    return W, hidden, drafts


@pytest.mark.parametrize("alpha", [0.0, 1.0])
def test_preblended_head_is_exact_at_alpha_0_and_1(alpha):
    # the blend is then one of the two bf16 rows itself: no rounding, same logits
    W, hidden, drafts = _preblend_case(42)
    a = orc.verify_head_preblended(W, hidden, drafts, 3, 2, alpha)
    b = orc.verify_head(W, hidden, drafts, 3, 2, alpha)
    np.testing.assert_array_equal(a["z"], b["z"])
    np.testing.assert_array_equal(a["argmax"], b["argmax"])
    np.testing.assert_array_equal(a["lse_fused"], b["lse_fused"])
    assert np.isnan(a["lse_orig"]).all() and np.isnan(a["ent_orig"]).all()


def test_preblended_head_within_the_bf16_rounding_bound():
    # |W b - z| <= sum_k |W_vk| |b_k - b*_k| with b* the exact blend, and
    # |b_k - b*_k| <= 2^-8 |b*_k| (float32 steps + one bf16 rounding)
    W, hidden, drafts = _preblend_case(43)
    alpha = 0.3
    a = orc.verify_head_preblended(W, hidden, drafts, 3, 2, alpha)
    b = orc.verify_head(W, hidden, drafts, 3, 2, alpha)
    h = orc.as_f64(hidden)
    oi = [orc.original_row(i) for i in range(1, 5)]
    ri = [orc.reflective_row(i, 3, 2) for i in range(1, 5)]
    exact = (1 - alpha) * h[:, oi, :] + alpha * h[:, ri, :]
    bound = np.einsum("vk,bik->biv", np.abs(orc.as_f64(W)), np.abs(exact)) * 2.0 ** -8
    diff = np.abs(a["z"] - b["z"])
    assert (diff <= bound).all()
    assert diff.max() > 0          # the rounding is real
    # every blended value is a bf16 number: a float32 whose low 16 bits are zero
    blend = orc.preblend_rows(hidden, 3, 2, alpha)
    assert not (np.asarray(blend, np.float32).view(np.uint32) & 0xFFFF).any()


def test_pins_catch_unrounded_blend(monkeypatch):
    real = orc.round_to_bf16
    monkeypatch.setattr(orc, "round_to_bf16", lambda x: np.asarray(x, np.float32))
    with pytest.raises(AssertionError):
        test_preblended_head_within_the_bf16_rounding_bound()
    monkeypatch.setattr(orc, "round_to_bf16", real)


def test_pins_catch_swapped_blend_weights(monkeypatch):
    real = orc.preblend_rows
    monkeypatch.setattr(orc, "preblend_rows", lambda h, g, R, a: real(h, g, R, 1.0 - a))
    with pytest.raises(AssertionError):
        test_preblended_head_is_exact_at_alpha_0_and_1(0.0)


# --------------------------------------------------------------------------
# Standard speculative verification, the baseline without reflection (Sec. 4)
# --------------------------------------------------------------------------

def test_standard_block_closed_form_and_first_segment():
    # the drafts alone at the positions after the context; they are the first
    # segment of the reflective block (Eq. 1)
    blk, pos = orc.pack_block_standard([[5, 6, 7], [1, 1, 2]], [10, 0])
    np.testing.assert_array_equal(blk, [[5, 6, 7], [1, 1, 2]])
    np.testing.assert_array_equal(pos, [[10, 11, 12], [0, 1, 2]])
    rng = np.random.default_rng(51)
    drafts = rng.integers(0, 100, (3, 4))
    full, fpos = orc.pack_block(drafts, np.array([9, 8], np.int32),
                                rng.integers(0, 100, (3, 4)), np.array([3, 7, 0]))
    s, spos = orc.pack_block_standard(drafts, np.array([3, 7, 0]))
    np.testing.assert_array_equal(full[:, :4], s)
    np.testing.assert_array_equal(fpos[:, :4], spos)


def test_standard_head_matches_torch_log_softmax():
    # o_i from hidden row i-1 (rows beyond gamma are not read), against
    # torch's fp64 matmul / log_softmax / logsumexp / argmax
    rng = np.random.default_rng(52)
    B, gamma, V, H = 3, 4, 300, 16
    W = rng.standard_normal((V, H)).astype(np.float32)
    hidden = rng.standard_normal((B, gamma + 2, H)).astype(np.float32)
    drafts = rng.integers(0, V, (B, gamma))
    r = orc.verify_head_standard(W, hidden, drafts, gamma)
    o = torch.from_numpy(hidden[:, :gamma + 1].astype(np.float64)) @ \
        torch.from_numpy(W.astype(np.float64)).T
    lsm = torch.log_softmax(o, dim=-1).numpy()
    np.testing.assert_allclose(r["lse_fused"], torch.logsumexp(o, dim=-1).numpy(), atol=1e-10)
    bi, ii = np.arange(B)[:, None], np.arange(gamma)[None, :]
    np.testing.assert_allclose(r["logp_fused"], lsm[bi, ii, drafts], atol=1e-10)
    np.testing.assert_array_equal(r["argmax"], torch.argmax(o, dim=-1).numpy())
    for f in ("lse_orig", "lse_refl", "logp_orig", "logp_refl", "ent_orig"):
        assert np.isnan(r[f]).all()


def test_standard_head_is_alpha_zero_of_the_reflective_head():
    # Eq. 2 at alpha = 0 is standard verification: with the same states in
    # rows 0..gamma, the reflective head's fused statistics equal these
    rng = np.random.default_rng(53)
    gamma, R = 3, 4
    W, hidden, drafts = _rand_head(rng, 2, gamma, R, 120, 8)
    r = orc.verify_head(W, hidden, drafts, gamma, R, 0.0)
    s = orc.verify_head_standard(W, hidden[:, :gamma + 1], drafts, gamma)
    for f in ("lse_fused", "logp_fused", "margin", "choice_gap"):
        np.testing.assert_allclose(s[f], r[f], atol=1e-10)
    np.testing.assert_array_equal(s["argmax"], r["argmax"])


def test_standard_step_attention_and_decisions():
    # the standard step's attention is the reflective block's first segment
    # (Sec. 3.1); at alpha = 0 both steps take the same decisions
    rng = np.random.default_rng(54)
    B, gamma, R, Hq, Hkv, D, V, H = 2, 3, 2, 4, 2, 8, 60, 8
    Lb = 2 * gamma + R
    q, kb, vb, kc, vc, ctx = _rand_attn(rng, B, Lb, Hq, Hkv, D, [4, 0], 20)
    W, hidden, _ = _rand_head(rng, B, gamma, R, V, H)
    choice = np.argmax(orc.as_f64(hidden[:, :gamma]) @ orc.as_f64(W).T, axis=-1)
    drafts = np.where(rng.random((B, gamma)) < 0.7, choice, rng.integers(0, V, (B, gamma)))
    full = orc.verify_step(W, hidden, q, kb, vb, kc, vc, ctx, drafts, np.array([1], np.int32),
                           rng.integers(0, V, (B, 1)), gamma, R, 0.0)
    std = orc.verify_step_standard(W, hidden[:, :gamma + 1], q[:, :gamma], kb[:, :gamma],
                                   vb[:, :gamma], kc, vc, ctx, drafts, gamma)
    np.testing.assert_array_equal(std["attn"], full["attn"][:, :gamma])
    for b, c in enumerate(ctx):
        np.testing.assert_array_equal(std["k_cache"][b, :, :c + gamma], full["k_cache"][b, :, :c + gamma])
    for f in ("accept_mask", "accepted_len", "next_token", "ctx_out"):
        np.testing.assert_array_equal(std[f], full[f])


def test_pins_catch_standard_row_off_by_one(monkeypatch):
    monkeypatch.setattr(orc, "original_row", lambda i: i)
    with pytest.raises(AssertionError):
        test_standard_head_matches_torch_log_softmax()


def test_pins_catch_standard_block_with_copy(monkeypatch):
    def with_copy(drafts, ctx_lens):
        d = np.asarray(drafts, np.int64)
        blk = np.concatenate([d, d], axis=1)
        pos = np.asarray(ctx_lens, np.int64)[:, None] + np.arange(blk.shape[1])
        return blk.astype(np.int32), pos.astype(np.int32)
    monkeypatch.setattr(orc, "pack_block_standard", with_copy)
    with pytest.raises(AssertionError):
        test_standard_block_closed_form_and_first_segment()


def test_pins_catch_inverse_cdf_slips(monkeypatch):
    # one token early (the last v whose cumulative weight is still below u * sum)
    real = orc.inverse_cdf_sample
    monkeypatch.setattr(orc, "inverse_cdf_sample", lambda w, u: max(0, real(w, u) - 1))
    with pytest.raises(AssertionError):
        test_inverse_cdf_sample_closed_forms()
    # u compared against unnormalised cumulative weights
    def unscaled(w, u):
        c = np.cumsum(np.asarray(w, np.float64))
        return int(min(np.searchsorted(c, u, side="right"), len(c) - 1))
    monkeypatch.setattr(orc, "inverse_cdf_sample", unscaled)
    with pytest.raises(AssertionError):
        test_inverse_cdf_sample_closed_forms()
