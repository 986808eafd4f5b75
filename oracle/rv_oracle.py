"""CPU oracle of the Reflective Verification verify step (arXiv 2505.18629).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference legs may import or run this module.  It
shares no code with the CUDA path (``paper_2505_18629_gb300``) and imports
nothing from it; the product never calls it.

Plain NumPy in float64: every bf16 (uint16 bit pattern) or fp32 input is first
widened exactly to float64, then each step below is its textbook definition.
No tiling, fusion or reordering beyond what the definitions state (the LM-head
product is computed a block of vocab rows at a time only to bound memory; each
logit is still one full dot product).

Notation follows the paper:
  * gamma  -- number of draft tokens x_1..x_gamma (Alg. 1)
  * template -- Prompt_reflection || Prefix_position (Eq. 1); R = |template|
  * reflective_draft = [x_1..x_gamma, template, x_1..x_gamma]  (Alg. 1, Eq. 1)
  * m = gamma + |template| + 1 (Alg. 1); shift_len = m - 1 (Eq. 2)
  * o_i (i = 1..gamma+1) original logits, o_{m+i-1} reflective logits
  * p_i = softmax((1-alpha) o_i + alpha o_{m+i-1})   (Eq. 2, Alg. 1)
  * exact-match verification with the greedy choice x^_i = argmax p_i
    (Alg. 2, read as "stop at the first mismatch"; see ``exact_match_accept``)
    or with sampled x^_i ~ softmax(z_i / T) (``sampled_exact_accept``)
  * typical acceptance (Alg. 3) and speculative sampling (Alg. 1)
  * the pre-blended head: z_i = W b_i with b_i the bf16-rounded blend of the
    two hidden states (``verify_head_preblended``; linearity of Eq. 2)
  * the pending-token block [t, x_1..x_gamma, template, x_1..x_gamma], whose
    first position is the last emitted token (``pack_block_pending``,
    ``verify_step_pending``)
  * standard speculative verification, the baseline the method is compared
    with (Sec. 4): block [x_1..x_gamma], p_i = softmax(o_i) from the gamma+1
    original rows alone (``pack_block_standard``, ``verify_head_standard``,
    ``verify_step_standard``)

Hidden-state rows: row 0 is the target's last hidden state after the prefix
(gives o_1, "M_p(prefix)" in Alg. 1); row r (1..Lb) follows block token r-1.
So o_i is row i-1 and its reflective partner o_{m+i-1} is row i-1+shift_len.

Every function below is pinned by tests in ``tests/test_oracle_pins.py``
against closed forms, library routines, invariants the paper states, or brute
force; none is "parity unpinned".
"""
from __future__ import annotations

import numpy as np

# --------------------------------------------------------------------------
# Widening
# --------------------------------------------------------------------------


def as_f64(x: np.ndarray) -> np.ndarray:
    """Exact float64 view of a bf16 bit pattern (uint16) or fp32/fp64 array."""
    x = np.asarray(x)
    if x.dtype == np.uint16:
        return (x.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    if x.dtype in (np.float32, np.float64):
        return x.astype(np.float64)
    raise TypeError(f"unsupported dtype {x.dtype}")


# --------------------------------------------------------------------------
# Block construction: Eq. 1, Alg. 1 ("Prepare the reflective draft template")
# --------------------------------------------------------------------------


def template(prompt_ids: np.ndarray, prefix_ids: np.ndarray) -> np.ndarray:
    """template = Prompt_reflection || Prefix_position (Eq. 1)."""
    return np.concatenate([np.asarray(prompt_ids, np.int64), np.asarray(prefix_ids, np.int64)])


def reflective_draft(drafts: np.ndarray, tmpl: np.ndarray) -> np.ndarray:
    """[x_1..x_gamma, template, x_1..x_gamma] (Alg. 1; Eq. 1 Draft_final)."""
    d = np.asarray(drafts, np.int64)
    return np.concatenate([d, np.asarray(tmpl, np.int64), d])


def m_index(gamma: int, R: int) -> int:
    """m = gamma + |template| + 1 (Alg. 1)."""
    return gamma + R + 1


def shift_len(gamma: int, R: int) -> int:
    """Positions between o_i and its reflective partner (Eq. 2): m - 1."""
    return m_index(gamma, R) - 1


def original_row(i: int) -> int:
    """Hidden row that yields o_i, i = 1..gamma+1 (row 0 = after the prefix)."""
    return i - 1


def reflective_row(i: int, gamma: int, R: int) -> int:
    """Hidden row that yields o_{m+i-1}, the reflective partner of o_i."""
    return original_row(i) + shift_len(gamma, R)


def pack_block(drafts, prompt_ids, prefix_ids, ctx_lens):
    """Verify block ids and position ids for every sequence.

    drafts [B, gamma], prompt_ids [n_prompt], prefix_ids [B, n_prefix],
    ctx_lens [B] -> block_ids [B, Lb], pos_ids [B, Lb] with Lb = 2 gamma + R.
    Position ids run on from the context (ctx, ctx+1, ...) for the whole block.
    """
    drafts = np.asarray(drafts, np.int64)
    B = drafts.shape[0]
    rows, pos = [], []
    for b in range(B):
        blk = reflective_draft(drafts[b], template(prompt_ids, prefix_ids[b]))
        rows.append(blk)
        pos.append(int(ctx_lens[b]) + np.arange(blk.shape[0], dtype=np.int64))
    return np.stack(rows).astype(np.int32), np.stack(pos).astype(np.int32)


def pack_block_pending(pending, drafts, prompt_ids, prefix_ids, ctx_lens):
    """Pending-token variant of the block: [t, x_1..x_gamma, template, x_1..x_gamma].

    The last emitted token t (pending[b]) has not gone through the target yet,
    so the block starts with it: its position is the first after the context,
    its final hidden state gives o_1 ("M_p(prefix)" in Alg. 1, with the
    prefix ending in t), and its key/value are appended with the block's.
    Returns block_ids, pos_ids [B, Lb + 1] (Lb = 2 gamma + R), positions
    ctx_b, ctx_b + 1, ...
    """
    pending = np.asarray(pending, np.int64)
    blk, _ = pack_block(drafts, prompt_ids, prefix_ids, ctx_lens)
    block = np.concatenate([pending[:, None], blk.astype(np.int64)], axis=1)
    pos = np.asarray(ctx_lens, np.int64)[:, None] + np.arange(block.shape[1], dtype=np.int64)
    return block.astype(np.int32), pos.astype(np.int32)


def pack_block_standard(drafts, ctx_lens):
    """Block of standard speculative verification (no reflection): the drafts
    alone, [x_1..x_gamma], at positions ctx_b, ctx_b + 1, ...
    Returns block_ids, pos_ids [B, gamma]."""
    drafts = np.asarray(drafts, np.int64)
    gamma = drafts.shape[1]
    pos = np.asarray(ctx_lens, np.int64)[:, None] + np.arange(gamma, dtype=np.int64)
    return drafts.astype(np.int32), pos.astype(np.int32)


# --------------------------------------------------------------------------
# One forward pass over the block: causal attention (Sec. 3.1)
# --------------------------------------------------------------------------


def verify_attention(q, k_blk, v_blk, k_cache, v_cache, ctx_lens):
    """Causal attention of the verify block against the KV cache (Sec. 3.1).

    q [B, Lb, Hq, D]; k_blk, v_blk [B, Lb, Hkv, D]; caches [B, Hkv, Cmax, D];
    ctx_lens [B].  Block query j of sequence b sits at position ctx_b + j and
    sees the cached keys 0..ctx_b-1 and block keys 0..j (unidirectional mask:
    the template and the copy cannot change what the first segment sees).
    Query head h reads key/value head h // (Hq / Hkv).

    Returns (out [B, Lb, Hq, D] float64, k_cache', v_cache') where the caches
    have the block's keys/values written at [ctx_b, ctx_b + Lb).
    """
    q, kb, vb = as_f64(q), as_f64(k_blk), as_f64(v_blk)
    kc, vc = as_f64(k_cache).copy(), as_f64(v_cache).copy()
    B, Lb, Hq, D = q.shape
    Hkv = kb.shape[2]
    G = Hq // Hkv
    out = np.zeros((B, Lb, Hq, D))
    scale = 1.0 / np.sqrt(D)
    for b in range(B):
        c = int(ctx_lens[b])
        for h in range(Hq):
            g = h // G
            keys = np.concatenate([kc[b, g, :c], kb[b, :, g]], axis=0)    # [c+Lb, D]
            vals = np.concatenate([vc[b, g, :c], vb[b, :, g]], axis=0)
            for j in range(Lb):
                n = c + j + 1                      # keys visible to query j
                s = keys[:n] @ q[b, j, h] * scale
                w = np.exp(s - s.max())
                w /= w.sum()
                out[b, j, h] = w @ vals[:n]
        kc[b, :, c:c + Lb] = kb[b].transpose(1, 0, 2)
        vc[b, :, c:c + Lb] = vb[b].transpose(1, 0, 2)
    return out, kc, vc


# --------------------------------------------------------------------------
# LM head, fusion (Eq. 2), log-softmax
# --------------------------------------------------------------------------


def head_logits(W, rows, block_rows: int = 8192) -> np.ndarray:
    """Logits W @ h for every row h: rows [N, H] -> [N, V] (no bias)."""
    rows = as_f64(rows)
    V = W.shape[0]
    out = np.empty((rows.shape[0], V))
    for v0 in range(0, V, block_rows):
        v1 = min(V, v0 + block_rows)
        out[:, v0:v1] = rows @ as_f64(W[v0:v1]).T
    return out


def logsumexp(x: np.ndarray, axis: int = -1) -> np.ndarray:
    """log(sum(exp(x))) along ``axis``, shifted by the max for range safety."""
    m = np.max(x, axis=axis, keepdims=True)
    return (m + np.log(np.sum(np.exp(x - m), axis=axis, keepdims=True))).squeeze(axis)


def entropy(logits: np.ndarray, axis: int = -1) -> np.ndarray:
    """Shannon entropy (nats) of softmax(logits): H = -sum_v p_v log p_v with
    log p_v = logits_v - logsumexp(logits).  Used by the entropy-based
    threshold of typical acceptance (Alg. 3)."""
    logits = np.asarray(logits, np.float64)
    logp = logits - np.expand_dims(logsumexp(logits, axis=axis), axis)
    p = np.exp(logp)
    return -np.sum(np.where(p > 0, p * logp, 0.0), axis=axis)


def fuse(o: np.ndarray, o_refl: np.ndarray, alpha: float) -> np.ndarray:
    """(1 - alpha) * o_i + alpha * o_{i + shift_len}  (Eq. 2, before softmax)."""
    return (1.0 - alpha) * o + alpha * o_refl


def greedy_choice(z: np.ndarray) -> np.ndarray:
    """argmax over the vocab (last axis); ties go to the lowest token id."""
    return np.argmax(z, axis=-1)


def verify_head(W, hidden, drafts, gamma: int, R: int, alpha: float):
    """LM head for the original and reflective rows, fused distribution p_i.

    W [V, H]; hidden [B, Lb+1, H]; drafts [B, gamma].
    For i = 1..gamma+1 (array index i-1):
      o_i = W h_{row i-1},  o_{m+i-1} = W h_{row i-1+shift_len},
      z_i = (1-alpha) o_i + alpha o_{m+i-1},  log p_i = z_i - logsumexp(z_i).
    Returns a dict of float64 / int64 arrays:
      lse_orig, lse_refl, lse_fused        [B, gamma+1]
      logp_fused, logp_orig, logp_refl     [B, gamma]  (at the draft x_i)
      argmax                               [B, gamma+1] (greedy x^_i)
      margin                               [B, gamma]  |z_i[x_i] - max_{v != x_i} z_i[v]|
      choice_gap                           [B, gamma+1] z_i[x^_i] - max_{v != x^_i} z_i[v]
                                           (how far the greedy choice is from a tie)
      ent_orig                             [B, gamma+1] entropy of softmax(o_i), the
                                           unfused original distribution (Alg. 3)
      z                                    [B, gamma+1, V] fused logits
    """
    hidden = as_f64(hidden)
    drafts = np.asarray(drafts, np.int64)
    B = hidden.shape[0]
    orig_idx = [original_row(i) for i in range(1, gamma + 2)]
    refl_idx = [reflective_row(i, gamma, R) for i in range(1, gamma + 2)]
    h_o = hidden[:, orig_idx, :].reshape(B * (gamma + 1), -1)
    h_r = hidden[:, refl_idx, :].reshape(B * (gamma + 1), -1)
    logits = head_logits(W, np.concatenate([h_o, h_r], axis=0))
    V = logits.shape[1]
    o = logits[:B * (gamma + 1)].reshape(B, gamma + 1, V)
    o_refl = logits[B * (gamma + 1):].reshape(B, gamma + 1, V)
    z = fuse(o, o_refl, alpha)
    lse_o, lse_r, lse_z = logsumexp(o), logsumexp(o_refl), logsumexp(z)
    bi = np.arange(B)[:, None]
    ii = np.arange(gamma)[None, :]
    zx = z[bi, ii, drafts]
    z_others = z[:, :gamma, :].copy()
    z_others[bi, ii, drafts] = -np.inf
    margin = np.abs(zx - z_others.max(axis=-1))
    choice = greedy_choice(z)
    z_rest = z.copy()
    np.put_along_axis(z_rest, choice[..., None], -np.inf, axis=-1)
    choice_gap = np.take_along_axis(z, choice[..., None], axis=-1)[..., 0] - z_rest.max(axis=-1)
    return dict(
        lse_orig=lse_o, lse_refl=lse_r, lse_fused=lse_z,
        logp_fused=zx - lse_z[:, :gamma],
        logp_orig=o[bi, ii, drafts] - lse_o[:, :gamma],
        logp_refl=o_refl[bi, ii, drafts] - lse_r[:, :gamma],
        argmax=choice, margin=margin, choice_gap=choice_gap, ent_orig=entropy(o), z=z,
    )


def round_to_bf16(x) -> np.ndarray:
    """float32 values rounded to the nearest bf16 (ties to even), as float32.

    bf16 keeps the top 16 bits of a float32: add half of the dropped range,
    plus one when the kept part is odd (ties to even), then truncate."""
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    keep_odd = (u >> 16) & 1
    r = ((u + 0x7FFF + keep_odd) >> 16) << 16
    return r.astype(np.uint32).view(np.float32)


def preblend_rows(hidden, gamma: int, R: int, alpha: float) -> np.ndarray:
    """The hidden state whose LM-head product is the fused logit vector.

    The head has no bias, so by linearity z_i = (1-a) W h + a W h' = W b_i
    with b_i = (1-a) h_{row i-1} + a h_{row i-1+shift_len} (Eq. 2).  A bf16
    LM head takes b_i in bf16: it is formed in float32 as
    fl((1-a) h) + fl(a h') (products rounded, then the sum rounded, no fused
    multiply-add) and then rounded to bf16.  That rounding is the variant's
    only difference from fusing the two logit vectors.
    Returns b [B, gamma+1, H] float32 (each value a bf16)."""
    h = as_f64(hidden).astype(np.float32)
    a = np.float32(alpha)
    beta = np.float32(np.float32(1.0) - a)
    orig_idx = [original_row(i) for i in range(1, gamma + 2)]
    refl_idx = [reflective_row(i, gamma, R) for i in range(1, gamma + 2)]
    blend = (beta * h[:, orig_idx, :]).astype(np.float32) + (a * h[:, refl_idx, :]).astype(np.float32)
    return round_to_bf16(blend.astype(np.float32))


def verify_head_preblended(W, hidden, drafts, gamma: int, R: int, alpha: float):
    """The fused distribution from pre-blended hidden states (a bf16 LM head).

    z_i = W b_i with b_i from ``preblend_rows``; everything derived from z
    (lse_fused, logp_fused, argmax, margin, choice_gap, z) as in
    ``verify_head``.  The unfused original / reflective distributions are not
    formed, so lse_orig, lse_refl, logp_orig, logp_refl and ent_orig are NaN."""
    drafts = np.asarray(drafts, np.int64)
    b = preblend_rows(hidden, gamma, R, alpha)
    B = b.shape[0]
    z = head_logits(W, b.reshape(B * (gamma + 1), -1)).reshape(B, gamma + 1, -1)
    lse_z = logsumexp(z)
    bi = np.arange(B)[:, None]
    ii = np.arange(gamma)[None, :]
    zx = z[bi, ii, drafts]
    z_others = z[:, :gamma, :].copy()
    z_others[bi, ii, drafts] = -np.inf
    margin = np.abs(zx - z_others.max(axis=-1))
    choice = greedy_choice(z)
    z_rest = z.copy()
    np.put_along_axis(z_rest, choice[..., None], -np.inf, axis=-1)
    choice_gap = np.take_along_axis(z, choice[..., None], axis=-1)[..., 0] - z_rest.max(axis=-1)
    nan1 = np.full((B, gamma + 1), np.nan)
    nan2 = np.full((B, gamma), np.nan)
    return dict(lse_orig=nan1, lse_refl=nan1.copy(), lse_fused=lse_z, logp_fused=zx - lse_z[:, :gamma],
                logp_orig=nan2, logp_refl=nan2.copy(), argmax=choice, margin=margin,
                choice_gap=choice_gap, ent_orig=nan1.copy(), z=z)


def verify_head_standard(W, hidden, drafts, gamma: int):
    """LM head of standard speculative verification: p_i = softmax(o_i).

    hidden [B, gamma+1, H] -- row 0 the state after the prefix, row i the
    state after x_i -- so o_i = W h_{row i-1} for i = 1..gamma+1, as in
    ``verify_head`` without the reflective rows (Eq. 2 at alpha = 0).  The
    result has ``verify_head``'s keys; the distribution is o's own, so its
    statistics sit in the fused fields (lse_fused, logp_fused, argmax,
    margin, choice_gap, z) and the original / reflective / entropy fields are
    NaN, as the single-distribution head leaves them."""
    hidden = as_f64(hidden)
    drafts = np.asarray(drafts, np.int64)
    B = hidden.shape[0]
    rows = [original_row(i) for i in range(1, gamma + 2)]
    o = head_logits(W, hidden[:, rows, :].reshape(B * (gamma + 1), -1)).reshape(B, gamma + 1, -1)
    lse = logsumexp(o)
    bi = np.arange(B)[:, None]
    ii = np.arange(gamma)[None, :]
    ox = o[bi, ii, drafts]
    o_others = o[:, :gamma, :].copy()
    o_others[bi, ii, drafts] = -np.inf
    margin = np.abs(ox - o_others.max(axis=-1))
    choice = greedy_choice(o)
    o_rest = o.copy()
    np.put_along_axis(o_rest, choice[..., None], -np.inf, axis=-1)
    choice_gap = np.take_along_axis(o, choice[..., None], axis=-1)[..., 0] - o_rest.max(axis=-1)
    nan1 = np.full((B, gamma + 1), np.nan)
    nan2 = np.full((B, gamma), np.nan)
    return dict(lse_orig=nan1, lse_refl=nan1.copy(), lse_fused=lse, logp_fused=ox - lse[:, :gamma],
                logp_orig=nan2, logp_refl=nan2.copy(), argmax=choice, margin=margin,
                choice_gap=choice_gap, ent_orig=nan1.copy(), z=o)


# --------------------------------------------------------------------------
# Exact-match verification (Alg. 2) with greedy x^_i, prefix, next token
# --------------------------------------------------------------------------


def exact_match_accept(drafts, choice):
    """Alg. 2 with x^_i = greedy choice of p_i.

    drafts [B, gamma], choice [B, gamma+1] (x^_1..x^_{gamma+1}).
    accept_i = (x_i == x^_i).  Alg. 2 prints the stopping set as the positions
    where x_i equals x^_i; the standard rule the paper says it keeps (Sec. 3.3:
    everything after the fusion is unchanged) stops at the first MISMATCH, so
    n = min({i-1 : x_i != x^_i} U {gamma}) and t = x^_{n+1}.
    Returns accept_mask [B, gamma] (uint8), n [B], next_token [B].
    """
    drafts = np.asarray(drafts, np.int64)
    choice = np.asarray(choice, np.int64)
    B, gamma = drafts.shape
    acc = (drafts == choice[:, :gamma])
    n = np.empty(B, np.int64)
    t = np.empty(B, np.int64)
    for b in range(B):
        stop = [i - 1 for i in range(1, gamma + 1) if not acc[b, i - 1]]
        n[b] = min(stop + [gamma])
        t[b] = choice[b, n[b]]
    return acc.astype(np.uint8), n, t


def typical_accept(drafts, logp_fused, ent_orig, choice, eps: float, delta: float):
    """Typical acceptance with Reflective Verification (Alg. 3).

    Position i keeps its draft when p_i(x_i) exceeds the entropy-based
    threshold min(eps, delta * exp(-H(p_original,i))), where p_i is the fused
    distribution of Eq. 2 and p_original,i = softmax(o_i) the unfused original
    one at the same position.  n is the number of leading kept drafts (the
    printed stopping set is read as "stop at the first draft that fails the
    threshold"), and the next token t is the greedy choice argmax p_{n+1}
    (the sampling temperature of Alg. 3 taken to 0, as for Alg. 2).

    Returns (accept_mask [B, gamma] bool, n [B], t [B], gap [B, gamma]) where
    gap = log p_i(x_i) - log threshold_i (the decision's distance in nats).
    """
    logp = np.asarray(logp_fused, np.float64)
    H = np.asarray(ent_orig, np.float64)[:, :logp.shape[1]]
    log_thr = np.minimum(np.log(eps), np.log(delta) - H)
    gap = logp - log_thr
    acc = gap > 0
    B, gamma = acc.shape
    n = np.full(B, gamma, np.int64)
    for b in range(B):
        for i in range(gamma):
            if not acc[b, i]:
                n[b] = i
                break
    t = np.asarray(choice, np.int64)[np.arange(B), n]
    return acc, n, t, gap


def inverse_cdf_sample(w: np.ndarray, u: float) -> int:
    """The token drawn from the distribution proportional to w >= 0 by one
    uniform u in [0, 1): the smallest v whose cumulative weight exceeds u * sum(w).
    If no cumulative weight exceeds it (u = 1, outside the domain), the draw is
    the last token of positive weight: a token of zero weight is never drawn."""
    w = np.asarray(w, np.float64)
    c = np.cumsum(w)
    v = int(np.searchsorted(c, u * c[-1], side="right"))
    if v >= len(w):
        pos = np.flatnonzero(w > 0)
        v = int(pos[-1]) if pos.size else len(w) - 1
    return v


def speculative_accept(drafts, z, q, r, u):
    """Speculative sampling with Reflective Verification (Alg. 1).

    drafts [B, gamma]; z [B, gamma+1, V] fused logits (p_i = softmax(z_i),
    Eq. 2); q [B, gamma, V] the draft model's distributions q_i; r [B, gamma]
    the uniforms r_i ~ U(0, 1); u [B] one more uniform per sequence for t.
    n is the number of leading drafts with r_i <= p_i(x_i) / q_i(x_i) (Alg. 1
    stops at the first i with r_i > p_i(x_i) / q_i(x_i)); t ~ p' with
    p' = norm(max(0, p_{n+1} - q_{n+1})) when n < gamma, else p' = p_{gamma+1},
    drawn by inverse CDF with u.

    Returns (accept_mask [B, gamma] bool, n [B], t [B], log_ratio [B, gamma],
    cdf_gap [B]) where log_ratio = log p_i(x_i) - log q_i(x_i) and cdf_gap is
    the distance of u from the nearest cumulative-weight boundary of p'
    (normalised), which bounds how close the draw of t was to a tie.
    """
    drafts = np.asarray(drafts, np.int64)
    z = np.asarray(z, np.float64)
    q = np.asarray(q, np.float64)
    r = np.asarray(r, np.float64)
    B, gamma = drafts.shape
    logp = z - logsumexp(z)[..., None]
    bi = np.arange(B)[:, None]
    ii = np.arange(gamma)[None, :]
    with np.errstate(divide="ignore"):
        log_ratio = logp[bi, ii, drafts] - np.log(q[bi, ii, drafts])
    acc = np.log(r) <= log_ratio
    n = np.full(B, gamma, np.int64)
    t = np.zeros(B, np.int64)
    cdf_gap = np.zeros(B)
    for b in range(B):
        for i in range(gamma):
            if not acc[b, i]:
                n[b] = i
                break
        p_next = np.exp(logp[b, n[b]])
        w = np.maximum(0.0, p_next - q[b, n[b]]) if n[b] < gamma else p_next
        if not w.sum() > 0:  # p_{n+1} <= q_{n+1} everywhere: only possible through rounding
            w = p_next
        t[b] = inverse_cdf_sample(w, float(u[b]))
        c = np.cumsum(w) / w.sum()
        cdf_gap[b] = np.min(np.abs(c - u[b]))
    return acc, n, t, log_ratio, cdf_gap


def sampled_exact_accept(drafts, z, temperature: float, u):
    """Exact-match verification with sampled target tokens (Alg. 2).

    drafts [B, gamma]; z [B, gamma+1, V] fused logits (Eq. 2); u [B, gamma+1]
    one uniform per position.  At sampling temperature T the target's token at
    position i is x^_i ~ softmax(z_i / T) (T = 1 gives p_i itself), drawn by
    inverse CDF with u[b, i].  Drafts are kept up to the first mismatch
    x_i != x^_i (the stopping set read as in ``exact_match_accept``), and the
    next token t ~ p_{n+1} is the draw x^_{n+1} already taken at that position:
    the emitted tokens [x_1..x_n, t] are then x^_1..x^_{n+1}, i.e. exactly what
    sampling the target alone would give, which makes the rule lossless
    (Sec. 4.1).  T -> 0 reduces to the greedy rule of ``exact_match_accept``.

    Returns (accept_mask [B, gamma] uint8, n [B], t [B], xhat [B, gamma+1],
    cdf_gap [B, gamma+1]) where cdf_gap is the distance of u from the nearest
    cumulative-weight boundary of softmax(z_i / T), which bounds how close
    each draw was to a tie.
    """
    z = np.asarray(z, np.float64)
    u = np.asarray(u, np.float64)
    B, G1, V = z.shape
    zt = z / float(temperature)
    p_t = np.exp(zt - logsumexp(zt)[..., None])
    xhat = np.zeros((B, G1), np.int64)
    cdf_gap = np.zeros((B, G1))
    for b in range(B):
        for i in range(G1):
            xhat[b, i] = inverse_cdf_sample(p_t[b, i], float(u[b, i]))
            c = np.cumsum(p_t[b, i]) / p_t[b, i].sum()
            cdf_gap[b, i] = np.min(np.abs(c - u[b, i]))
    acc, n, t = exact_match_accept(drafts, xhat)
    return acc, n, t, xhat, cdf_gap


def typical_accept_sampled(drafts, logp_fused, ent_orig, z, eps: float, delta: float,
                           temperature: float, u):
    """Typical acceptance (Alg. 3) with the next token sampled at temperature T.

    The kept drafts and n are those of ``typical_accept`` (the entropy
    threshold on the fused distribution, Eq. 2); the next token is drawn as
    Alg. 3 states, t ~ p_{n+1}, at sampling temperature T: the inverse CDF of
    softmax(z_{n+1} / T) at the uniform u[b, n] (one uniform per position,
    [B, gamma+1], as for ``sampled_exact_accept``).  T -> 0 gives the greedy t
    of ``typical_accept``.

    Returns (accept_mask [B, gamma] bool, n [B], t [B], gap [B, gamma],
    cdf_gap [B]) with gap as in ``typical_accept`` and cdf_gap the distance of
    u[b, n] from the nearest cumulative-weight boundary of the draw.
    """
    z = np.asarray(z, np.float64)
    u = np.asarray(u, np.float64)
    B = z.shape[0]
    acc, n, _, gap = typical_accept(drafts, logp_fused, ent_orig,
                                    np.zeros(z.shape[:2], np.int64), eps, delta)
    t = np.zeros(B, np.int64)
    cdf_gap = np.zeros(B)
    for b in range(B):
        zt = z[b, n[b]] / float(temperature)
        w = np.exp(zt - zt.max())
        t[b] = inverse_cdf_sample(w, float(u[b, n[b]]))
        c = np.cumsum(w) / w.sum()
        cdf_gap[b] = np.min(np.abs(c - u[b, n[b]]))
    return acc, n, t, gap, cdf_gap


def verify_step(inp_W, hidden, q, k_blk, v_blk, k_cache, v_cache, ctx_lens,
                drafts, prompt_ids, prefix_ids, gamma: int, R: int, alpha: float):
    """One whole verify step: pack, attention, head + fusion, accept, prefix.

    Returns a dict with every intermediate the CUDA path exposes.  The new
    context length is ctx + n: of the block's keys/values only the accepted
    drafts of the first segment stay valid (the template and copy are pruned,
    Sec. 3.1).
    """
    block_ids, pos_ids = pack_block(drafts, prompt_ids, prefix_ids, ctx_lens)
    attn, kc, vc = verify_attention(q, k_blk, v_blk, k_cache, v_cache, ctx_lens)
    head = verify_head(inp_W, hidden, drafts, gamma, R, alpha)
    acc, n, t = exact_match_accept(drafts, head["argmax"])
    return dict(block_ids=block_ids, pos_ids=pos_ids, attn=attn, k_cache=kc, v_cache=vc,
                accept_mask=acc, accepted_len=n, next_token=t,
                ctx_out=np.asarray(ctx_lens, np.int64) + n, **head)


def verify_step_pending(inp_W, hidden, q, k_blk, v_blk, k_cache, v_cache, ctx_lens, pending,
                        drafts, prompt_ids, prefix_ids, gamma: int, R: int, alpha: float):
    """The verify step with the pending-token block [t, x_1..x_gamma, template,
    x_1..x_gamma] (Lb + 1 = 2 gamma + R + 1 positions after the context).

    Hidden row 0 is the pending token's (it gives o_1), so the head's rows are
    those of ``verify_head`` unchanged: original rows 0..gamma, reflective
    rows gamma+R..2 gamma+R.  The attention covers the Lb + 1 block positions
    and appends all their keys/values.  Of those, t and the n accepted drafts
    stay in the context: the new length is ctx + 1 + n (the template, the
    copy and the rejected drafts are pruned by length, Sec. 3.1).
    """
    block_ids, pos_ids = pack_block_pending(pending, drafts, prompt_ids, prefix_ids, ctx_lens)
    attn, kc, vc = verify_attention(q, k_blk, v_blk, k_cache, v_cache, ctx_lens)
    head = verify_head(inp_W, hidden, drafts, gamma, R, alpha)
    acc, n, t = exact_match_accept(drafts, head["argmax"])
    return dict(block_ids=block_ids, pos_ids=pos_ids, attn=attn, k_cache=kc, v_cache=vc,
                accept_mask=acc, accepted_len=n, next_token=t,
                ctx_out=np.asarray(ctx_lens, np.int64) + 1 + n, **head)


def verify_step_standard(inp_W, hidden, q, k_blk, v_blk, k_cache, v_cache, ctx_lens, drafts,
                         gamma: int):
    """One step of standard speculative verification, the method's baseline:
    block [x_1..x_gamma] (``pack_block_standard``), causal attention over its
    gamma positions, p_i = softmax(o_i) from hidden [B, gamma+1, H]
    (``verify_head_standard``), exact match (Alg. 2), new context ctx + n
    (the rejected drafts' keys/values are dropped by length)."""
    block_ids, pos_ids = pack_block_standard(drafts, ctx_lens)
    attn, kc, vc = verify_attention(q, k_blk, v_blk, k_cache, v_cache, ctx_lens)
    head = verify_head_standard(inp_W, hidden, drafts, gamma)
    acc, n, t = exact_match_accept(drafts, head["argmax"])
    return dict(block_ids=block_ids, pos_ids=pos_ids, attn=attn, k_cache=kc, v_cache=vc,
                accept_mask=acc, accepted_len=n, next_token=t,
                ctx_out=np.asarray(ctx_lens, np.int64) + n, **head)
