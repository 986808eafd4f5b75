"""Helpers of the GPU parity tests: move a synthetic step to the device, run
the CUDA path through the C ABI, and compare against the oracle with the
tolerances of the verify step:

* accept decisions, accepted lengths and next tokens bit-exact, except where
  the oracle's decision margin is below MARGIN_EPS (counted and reported);
* log-probabilities / log-sum-exps within LOGP_ATOL absolute;
* attention outputs within ATTN_RTOL relative (to |ref| + the row's RMS);
* KV-cache append bit-exact.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch

import oracle.rv_oracle as orc
from paper_2505_18629_gb300 import synth

MARGIN_EPS = 1e-3
LOGP_ATOL = 2e-3
ATTN_RTOL = 1e-2


def to_dev(x: np.ndarray, dev="cuda") -> torch.Tensor:
    """numpy (uint16 bf16 bits / float32 / int32) -> contiguous device tensor."""
    if x.dtype == np.uint16:
        return torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).to(dev).contiguous()
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev).contiguous()


def to_np(t: torch.Tensor) -> np.ndarray:
    if t.dtype == torch.bfloat16:
        return t.cpu().view(torch.int16).numpy().view(np.uint16)
    return t.cpu().numpy()


def oracle_choice(inp: synth.VerifyInputs, alpha: float, seqs=None) -> np.ndarray:
    """The oracle's fused greedy choice x^_1..x^_gamma for (a sample of) the sequences."""
    wl = inp.wl
    seqs = np.arange(wl.B) if seqs is None else np.asarray(seqs)
    dummy = np.zeros((len(seqs), wl.gamma), np.int64)
    return orc.verify_head(inp.W, inp.hidden[seqs], dummy, wl.gamma, wl.R, alpha)["argmax"][:, :wl.gamma]


def oracle_drafts(inp: synth.VerifyInputs, alpha: float, seqs=None) -> np.ndarray:
    """Drafts = the oracle's fused greedy choice with probability p, else random.

    With `seqs`, only those sequences get the target's choice; the others keep
    their random alternative ids (they are not compared)."""
    wl = inp.wl
    choice = inp.draft_alt.copy()
    idx = np.arange(wl.B) if seqs is None else np.asarray(seqs)
    choice[idx] = oracle_choice(inp, alpha, idx)
    return synth.make_drafts(inp, choice)


@dataclasses.dataclass
class GpuRun:
    attn: np.ndarray
    k_cache: np.ndarray
    v_cache: np.ndarray
    scores: np.ndarray
    argmax: np.ndarray
    margin: np.ndarray
    accept_mask: np.ndarray
    accepted_len: np.ndarray
    next_token: np.ndarray
    ctx_out: np.ndarray
    block_ids: np.ndarray
    pos_ids: np.ndarray
    status: int


def make_handle(wl: synth.Workload, max_batch=None, max_gamma=None, max_template=None):
    from paper_2505_18629_gb300 import rv
    return rv.rv_create(wl.H, wl.V, wl.Hq, wl.Hkv, wl.D, max_batch or wl.B,
                        max_gamma or wl.gamma, max_template or wl.R, wl.capacity,
                        rv.RV_DTYPE_BF16 if wl.dtype == "bf16" else rv.RV_DTYPE_F32)


def run_gpu(inp: synth.VerifyInputs, drafts: np.ndarray, alpha: float, h=None) -> GpuRun:
    from paper_2505_18629_gb300 import rv
    wl = inp.wl
    own = h is None
    if own:
        h = make_handle(wl)
    B, g, R = wl.B, wl.gamma, wl.R
    W = to_dev(inp.W)
    hidden = to_dev(inp.hidden)
    q, kb, vb = to_dev(inp.q), to_dev(inp.k_blk), to_dev(inp.v_blk)
    kc, vc = to_dev(inp.k_cache), to_dev(inp.v_cache)
    ctx = to_dev(inp.ctx_lens.astype(np.int32))
    d = to_dev(drafts.astype(np.int32))
    prompt = to_dev(inp.prompt_ids.astype(np.int32)) if inp.prompt_ids.size else None
    prefix = to_dev(inp.prefix_ids.astype(np.int32))
    Lb = wl.Lb
    block = torch.full((B, Lb), -7, dtype=torch.int32, device="cuda")
    pos = torch.full((B, Lb), -7, dtype=torch.int32, device="cuda")
    attn = torch.zeros_like(q)
    scores = torch.full((B, g + 1, rv.RV_NSCORES), float("nan"), device="cuda")
    argmax = torch.full((B, g + 1), -7, dtype=torch.int32, device="cuda")
    margin = torch.full((B, g), float("nan"), device="cuda")
    acc = torch.full((B, g), 7, dtype=torch.uint8, device="cuda")
    alen = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    nxt = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    ctx_out = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    rv.rv_verify_step(h, q, kb, vb, kc, vc, hidden, W, d, prompt, prefix, ctx, alpha, block, pos,
                      attn, scores, argmax, margin, acc, alen, nxt, ctx_out)
    status = rv.rv_read_status(h)
    out = GpuRun(to_np(attn), to_np(kc), to_np(vc), to_np(scores), to_np(argmax), to_np(margin),
                 to_np(acc), to_np(alen), to_np(nxt), to_np(ctx_out), to_np(block), to_np(pos),
                 status)
    if own:
        h.close()
    return out


def attn_close(gpu_bits: np.ndarray, ref: np.ndarray, rtol=ATTN_RTOL):
    g = orc.as_f64(gpu_bits)
    rms = np.sqrt(np.mean(ref ** 2, axis=-1, keepdims=True))
    err = np.abs(g - ref)
    bound = rtol * (np.abs(ref) + rms)
    bad = err > bound
    return (not bad.any()), float((err / (np.abs(ref) + rms)).max()), int(bad.sum())


@dataclasses.dataclass
class Report:
    n_positions: int
    n_low_margin: int
    n_mask_mismatch: int
    n_seq_mismatch_excused: int
    max_lse_err: float
    max_logp_err: float
    max_margin_err: float
    attn_max_rel: float


def _err(gpu_vals: np.ndarray, ref_vals: np.ndarray) -> float:
    """Largest absolute difference; a field the oracle leaves NaN (the
    pre-blended head's original / reflective statistics) must be NaN on the
    GPU too and contributes 0."""
    if np.isnan(ref_vals).all():
        assert np.isnan(gpu_vals).all(), "a field without a value is not NaN"
        return 0.0
    return float(np.abs(gpu_vals - ref_vals).max())


def compare(inp: synth.VerifyInputs, drafts, alpha, ref: dict, gpu: GpuRun, check_attn=True,
            seqs=None, pending=None, standard=False) -> Report:
    """Assert GPU == oracle under the tolerances above; `seqs` restricts to sampled sequences.
    `pending` [B]: the step ran over the pending-token block [t, x, template, x].
    `standard`: standard verification's block [x] (or [t, x])."""
    wl = inp.wl
    g = wl.gamma
    seqs = np.arange(wl.B) if seqs is None else np.asarray(seqs)
    lead = 0 if pending is None else 1
    Lb = g if standard else wl.Lb
    assert gpu.status == 0, f"device status 0x{gpu.status:x}"
    # ---- pack
    if standard:
        d = drafts[seqs] if pending is None else np.concatenate(
            [np.asarray(pending)[seqs, None], drafts[seqs]], axis=1)
        blk, pos = orc.pack_block_standard(d, inp.ctx_lens[seqs])
    elif pending is None:
        blk, pos = orc.pack_block(drafts[seqs], inp.prompt_ids, inp.prefix_ids[seqs],
                                  inp.ctx_lens[seqs])
    else:
        blk, pos = orc.pack_block_pending(pending[seqs], drafts[seqs], inp.prompt_ids,
                                          inp.prefix_ids[seqs], inp.ctx_lens[seqs])
    np.testing.assert_array_equal(gpu.block_ids[seqs], blk)
    np.testing.assert_array_equal(gpu.pos_ids[seqs], pos)
    # ---- attention + cache append
    amax = 0.0
    if check_attn:
        ok, amax, nbad = attn_close(gpu.attn[seqs], ref["attn"])
        assert ok, f"attention: {nbad} elements beyond {ATTN_RTOL} relative (max {amax:.3g})"
        for k, b in enumerate(seqs):
            c = int(inp.ctx_lens[b]) + Lb + lead
            np.testing.assert_array_equal(gpu.k_cache[b, :, :c],
                                          _bits_like(ref["k_cache"][k, :, :c], gpu.k_cache))
            np.testing.assert_array_equal(gpu.v_cache[b, :, :c],
                                          _bits_like(ref["v_cache"][k, :, :c], gpu.v_cache))
    # ---- head scores
    sc = gpu.scores[seqs].astype(np.float64)
    lse_err = max(_err(sc[..., 0], ref["lse_orig"]), _err(sc[..., 1], ref["lse_refl"]),
                  _err(sc[..., 2], ref["lse_fused"]))
    assert lse_err <= LOGP_ATOL, f"lse error {lse_err}"
    logp_err = max(_err(sc[:, :g, 3], ref["logp_fused"]), _err(sc[:, :g, 4], ref["logp_orig"]),
                   _err(sc[:, :g, 5], ref["logp_refl"]))
    assert logp_err <= LOGP_ATOL, f"log-prob error {logp_err}"
    assert np.isnan(sc[:, g, 3:6]).all()
    ent_err = _err(sc[..., 6], ref["ent_orig"])
    assert ent_err <= LOGP_ATOL, f"entropy error {ent_err}"
    m_err = np.abs(gpu.margin[seqs].astype(np.float64) - ref["margin"]).max()
    assert m_err <= LOGP_ATOL, f"margin error {m_err}"
    if "typical_gap" in ref:
        return _compare_typical(inp, ref, gpu, seqs, lse_err, logp_err, m_err, amax)
    # ---- decisions with the margin rule
    low = ref["margin"] < MARGIN_EPS                       # [S, gamma]
    low_choice = ref["choice_gap"] < MARGIN_EPS            # [S, gamma+1]
    am_ok = (gpu.argmax[seqs] == ref["argmax"]) | low_choice
    assert am_ok.all(), "argmax differs at a position with a clear choice"
    mask_mismatch = (gpu.accept_mask[seqs] != ref["accept_mask"])
    assert not (mask_mismatch & ~low).any(), "accept mask differs at a clear decision"
    excused = 0
    for k, b in enumerate(seqs):
        n_ref = int(ref["accepted_len"][k])
        same = (gpu.accepted_len[b] == n_ref and gpu.next_token[b] == ref["next_token"][k])
        if not same:
            lim = min(n_ref + 1, g)
            assert low[k, :lim].any() or low_choice[k, min(n_ref, g)], \
                f"sequence {b}: accepted {gpu.accepted_len[b]} vs {n_ref} without a close decision"
            excused += 1
        assert gpu.ctx_out[b] == inp.ctx_lens[b] + lead + gpu.accepted_len[b]
        n = int(gpu.accepted_len[b])
        assert gpu.accept_mask[b, :n].all() and (n == g or gpu.accept_mask[b, n] == 0)
        assert gpu.next_token[b] == gpu.argmax[b, n]
    return Report(int(low.size), int(low.sum()), int(mask_mismatch.sum()), excused,
                  float(lse_err), float(logp_err), float(m_err), amax)


def compare_head(ref: dict, scores: np.ndarray, argmax: np.ndarray, margin: np.ndarray,
                 gamma: int) -> Report:
    """LM-head outputs (scores, argmax, margin of rv_verify_head) against the
    oracle's verify_head on the same sequences: statistics within LOGP_ATOL,
    the choice bit-exact except where the oracle's choice gap is below
    MARGIN_EPS (counted)."""
    g = gamma
    sc = scores.astype(np.float64)
    lse_err = max(_err(sc[..., 0], ref["lse_orig"]), _err(sc[..., 1], ref["lse_refl"]),
                  _err(sc[..., 2], ref["lse_fused"]))
    assert lse_err <= LOGP_ATOL, f"lse error {lse_err}"
    logp_err = max(_err(sc[:, :g, 3], ref["logp_fused"]), _err(sc[:, :g, 4], ref["logp_orig"]),
                   _err(sc[:, :g, 5], ref["logp_refl"]))
    assert logp_err <= LOGP_ATOL, f"log-prob error {logp_err}"
    assert np.isnan(sc[:, g, 3:6]).all()                  # no draft at the bonus position
    ent_err = _err(sc[..., 6], ref["ent_orig"])
    assert ent_err <= LOGP_ATOL, f"entropy error {ent_err}"
    m_err = float(np.abs(margin.astype(np.float64) - ref["margin"]).max())
    assert m_err <= LOGP_ATOL, f"margin error {m_err}"
    low_choice = ref["choice_gap"] < MARGIN_EPS
    assert ((argmax == ref["argmax"]) | low_choice).all(), \
        "argmax differs at a position with a clear choice"
    return Report(int(low_choice.size), int(low_choice.sum()), 0, 0, float(lse_err),
                  float(logp_err), m_err, 0.0)


def _compare_typical(inp, ref, gpu, seqs, lse_err, logp_err, m_err, amax) -> Report:
    """Typical acceptance (Alg. 3): decisions bit-exact except where the oracle's
    log p_i(x_i) is within MARGIN_EPS of the log threshold (counted); n and t may
    differ only past such a position; t is the greedy choice at n+1."""
    wl = inp.wl
    g = wl.gamma
    low = np.abs(ref["typical_gap"]) < MARGIN_EPS
    low_choice = ref["choice_gap"] < MARGIN_EPS
    am_ok = (gpu.argmax[seqs] == ref["argmax"]) | low_choice
    assert am_ok.all(), "argmax differs at a position with a clear choice"
    mism = gpu.accept_mask[seqs] != ref["accept_mask"]
    assert not (mism & ~low).any(), "typical accept mask differs at a clear decision"
    excused = 0
    for k, b in enumerate(seqs):
        n_ref = int(ref["accepted_len"][k])
        same = gpu.accepted_len[b] == n_ref and gpu.next_token[b] == ref["next_token"][k]
        if not same:
            lim = min(n_ref + 1, g)
            assert low[k, :lim].any() or low_choice[k, min(n_ref, g)], \
                f"sequence {b}: accepted {gpu.accepted_len[b]} vs {n_ref} without a close decision"
            excused += 1
        assert gpu.ctx_out[b] == inp.ctx_lens[b] + gpu.accepted_len[b]
        n = int(gpu.accepted_len[b])
        assert gpu.accept_mask[b, :n].all() and (n == g or gpu.accept_mask[b, n] == 0)
        assert gpu.next_token[b] == gpu.argmax[b, n]
    return Report(int(low.size), int(low.sum()), int(mism.sum()), excused, float(lse_err),
                  float(logp_err), float(m_err), amax)


def oracle_typical(inp, drafts, alpha, eps, delta, seqs=None, with_attn=True):
    """Oracle verify step with the typical acceptance of Alg. 3."""
    ref = oracle_step(inp, drafts, alpha, seqs=seqs, with_attn=with_attn)
    wl = inp.wl
    seqs = np.arange(wl.B) if seqs is None else np.asarray(seqs)
    acc, n, t, gap = orc.typical_accept(drafts[seqs], ref["logp_fused"], ref["ent_orig"],
                                        ref["argmax"], eps, delta)
    ref.update(accept_mask=acc.astype(np.uint8), accepted_len=n, next_token=t, typical_gap=gap)
    return ref


def _bits_like(ref_f64: np.ndarray, like: np.ndarray) -> np.ndarray:
    """The oracle's cache (exact widening of the inputs) back in the input encoding."""
    if like.dtype == np.uint16:
        return synth.to_bf16_bits(ref_f64.astype(np.float32))
    return ref_f64.astype(like.dtype)


def oracle_step(inp: synth.VerifyInputs, drafts, alpha, seqs=None, with_attn=True,
                preblended=False):
    """Oracle verify step on all or on a sample of the sequences
    (`preblended`: the head on the blended hidden states)."""
    wl = inp.wl
    seqs = np.arange(wl.B) if seqs is None else np.asarray(seqs)
    head_fn = orc.verify_head_preblended if preblended else orc.verify_head
    head = head_fn(inp.W, inp.hidden[seqs], drafts[seqs], wl.gamma, wl.R, alpha)
    acc, n, t = orc.exact_match_accept(drafts[seqs], head["argmax"])
    ref = dict(head, accept_mask=acc, accepted_len=n, next_token=t)
    ref.pop("z")
    if with_attn:
        out, kc, vc = orc.verify_attention(inp.q[seqs], inp.k_blk[seqs], inp.v_blk[seqs],
                                           inp.k_cache[seqs], inp.v_cache[seqs],
                                           inp.ctx_lens[seqs])
        ref.update(attn=out, k_cache=kc, v_cache=vc)
    return ref
