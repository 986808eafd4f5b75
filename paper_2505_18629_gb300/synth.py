"""Seeded synthetic inputs for the Reflective Verification verify step.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic (no attention, no logits, no softmax, no acceptance rule).
Both the CUDA path (tests, bench) and the CPU oracle take their inputs from it.

The paper's workloads (MT-Bench / GSM8K / HumanEval decoding with Llama-3.x
1B/8B/70B, Sec. 4.1 and Table 4) need datasets and trained weights that are not
available, so seeded Gaussian tensors with the same shapes stand in:

* LM-head weight ``W`` [V, H], hidden states [B, Lb+1, H];
* one attention layer: post-RoPE queries [B, Lb, Hq, D], the block's keys and
  values [B, Lb, Hkv, D], and a KV cache [B, Hkv, Cmax, D] per tensor;
* token ids: reflection prompt, the last ``n_prefix`` context tokens
  (Prefix_position of Eq. 1) and the draft tokens.

Drafts are "the target's choice with probability p, else a random id".  The
target's choice depends on the method's arithmetic, so this module only draws
the two random parts (``draft_keep`` Bernoulli(p) and ``draft_alt`` ids) and
``make_drafts`` combines them with an argmax that the caller supplies.

Draw order (PCG64, one seed per workload): W, hidden, Q, K_blk, V_blk, K cache,
V cache, ctx_lens, prompt ids, prefix ids, draft_keep, draft_alt.

bf16 tensors are returned as ``numpy.uint16`` bit patterns (round-to-nearest-
even from float32, done by torch); fp32 workloads return ``numpy.float32``.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np

__all__ = [
    "Workload", "WORKLOADS", "sweep_workloads", "VerifyInputs", "generate",
    "make_drafts", "to_bf16_bits", "bf16_bits_to_f32", "workload",
]

# Prefix_position length of Eq. 1: Table 4 uses 4 for every setting.
DEFAULT_PREFIX_LEN = 4
# Weight of the reflective logits, Table 4 (0.3 in every setting).
DEFAULT_ALPHA = 0.3

_ROW_CHUNK = 8192  # rows drawn per RNG call for the big weight (bounds memory)


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and value recipe of one synthetic verify step."""
    name: str
    B: int                    # sequences in the batch
    gamma: int                # draft tokens per sequence
    R: int                    # template length |template| = prompt + prefix
    ctx: tuple                # (lo, hi) inclusive context length range per sequence
    H: int                    # hidden size
    Hq: int                   # query heads
    Hkv: int                  # key/value heads
    D: int                    # head dim
    V: int                    # vocab size
    dtype: str                # "bf16" or "f32"
    p_argmax: float           # probability that a draft equals the target's choice
    draft_dist: str = "uniform"   # distribution of non-target drafts: uniform | zipf1.1
    value_std: float = 1.0    # std of Q/K/V/cache entries
    hidden_rms1: bool = True  # hidden rows N(0,1) rescaled to RMS 1 (else N(0, value_std))
    w_std: float = 0.02
    n_prefix: int = DEFAULT_PREFIX_LEN
    seed: int = 0
    cmax: Optional[int] = None  # cache capacity; default max ctx + Lb

    @property
    def Lb(self) -> int:
        """Verify block length: drafts + template + drafts (Eq. 1)."""
        return 2 * self.gamma + self.R

    @property
    def Lh(self) -> int:
        """Hidden rows per sequence: the last context position plus the block."""
        return self.Lb + 1

    @property
    def n_prompt(self) -> int:
        return self.R - min(self.n_prefix, self.R)

    @property
    def n_prefix_eff(self) -> int:
        return min(self.n_prefix, self.R)

    @property
    def capacity(self) -> int:
        return self.cmax if self.cmax is not None else self.ctx[1] + self.Lb

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


WORKLOADS = {
    # Tiny step the oracle finishes instantly: B=1, gamma=4, template 4 (Lb=12),
    # ctx 64, H=256, 4/4 heads of 64, V=4096, fp32, everything N(0, 0.02).
    "tiny": Workload("tiny", B=1, gamma=4, R=4, ctx=(64, 64), H=256, Hq=4, Hkv=4, D=64,
                     V=4096, dtype="f32", p_argmax=0.7, value_std=0.02, hidden_rms1=False,
                     seed=0),
    # Llama-3-8B-shaped step at batch 1 (gamma=5, template 8, ctx 2048).
    "llama3-8b-b1": Workload("llama3-8b-b1", B=1, gamma=5, R=8, ctx=(2048, 2048), H=4096,
                             Hq=32, Hkv=8, D=128, V=128256, dtype="bf16", p_argmax=0.7,
                             seed=1),
    # 8B-shaped step at batch 16, ctx ~ U[512, 4096], Zipf(1.1) non-target drafts.
    "llama3-8b-b16": Workload("llama3-8b-b16", B=16, gamma=8, R=8, ctx=(512, 4096), H=4096,
                              Hq=32, Hkv=8, D=128, V=128256, dtype="bf16", p_argmax=0.6,
                              draft_dist="zipf1.1", seed=2),
    # Llama-3-70B-shaped step at batch 32.
    "llama3-70b-b32": Workload("llama3-70b-b32", B=32, gamma=6, R=8, ctx=(4096, 4096), H=8192,
                               Hq=64, Hkv=8, D=128, V=128256, dtype="bf16", p_argmax=0.5,
                               seed=3),
}


def sweep_workloads():
    """8B-shaped sweep: B in {1,4,16,64} x gamma in {2,4,8} x ctx in {1024,8192}."""
    out = []
    k = 0
    for B in (1, 4, 16, 64):
        for g in (2, 4, 8):
            for c in (1024, 8192):
                out.append(Workload(f"sweep-b{B}-g{g}-c{c}", B=B, gamma=g, R=8, ctx=(c, c),
                                    H=4096, Hq=32, Hkv=8, D=128, V=128256, dtype="bf16",
                                    p_argmax=0.7, seed=100 + k))
                k += 1
    return out


def workload(name: str) -> Workload:
    if name in WORKLOADS:
        return WORKLOADS[name]
    for w in sweep_workloads():
        if w.name == name:
            return w
    raise KeyError(name)


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round-to-nearest-even (torch)."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> float32 (exact widening)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


@dataclasses.dataclass
class VerifyInputs:
    """One synthetic verify step.  bf16 tensors are uint16 bit patterns."""
    wl: Workload
    W: np.ndarray          # [V, H]
    hidden: np.ndarray     # [B, Lb+1, H]
    q: np.ndarray          # [B, Lb, Hq, D]
    k_blk: np.ndarray      # [B, Lb, Hkv, D]
    v_blk: np.ndarray      # [B, Lb, Hkv, D]
    k_cache: np.ndarray    # [B, Hkv, Cmax, D]
    v_cache: np.ndarray    # [B, Hkv, Cmax, D]
    ctx_lens: np.ndarray   # [B] int32
    prompt_ids: np.ndarray  # [R - n_prefix] int32
    prefix_ids: np.ndarray  # [B, n_prefix] int32  (last context tokens)
    draft_keep: np.ndarray  # [B, gamma] bool
    draft_alt: np.ndarray   # [B, gamma] int32

    @property
    def is_bf16(self) -> bool:
        return self.wl.dtype == "bf16"


def _values(rng, shape, std, bf16):
    x = rng.standard_normal(shape, dtype=np.float32)
    if std != 1.0:
        x *= np.float32(std)
    return to_bf16_bits(x) if bf16 else x


def _big_weight(rng, V, H, std, bf16):
    out = np.empty((V, H), dtype=np.uint16 if bf16 else np.float32)
    for r0 in range(0, V, _ROW_CHUNK):
        r1 = min(V, r0 + _ROW_CHUNK)
        out[r0:r1] = _values(rng, (r1 - r0, H), std, bf16)
    return out


def _zipf_ids(rng, n, V, s=1.1):
    ranks = np.arange(1, V + 1, dtype=np.float64)
    p = ranks ** (-s)
    p /= p.sum()
    return rng.choice(V, size=n, p=p).astype(np.int32)


def generate(wl: Workload, *, with_weight: bool = True, with_cache: bool = True) -> VerifyInputs:
    """Draw every input of one verify step from ``wl.seed`` (fixed draw order).

    ``with_weight=False`` / ``with_cache=False`` skip the two large tensors
    (their draws are then absent, so later draws differ: only use this for
    callers that never compare against a full draw).
    """
    rng = np.random.Generator(np.random.PCG64(wl.seed))
    bf16 = wl.dtype == "bf16"
    B, Lb, Lh = wl.B, wl.Lb, wl.Lh
    if with_weight:
        W = _big_weight(rng, wl.V, wl.H, wl.w_std, bf16)
    else:
        W = np.zeros((0, wl.H), dtype=np.uint16 if bf16 else np.float32)
    if wl.hidden_rms1:
        h = rng.standard_normal((B, Lh, wl.H), dtype=np.float32)
        rms = np.sqrt(np.mean(h.astype(np.float64) ** 2, axis=-1, keepdims=True))
        h = (h / rms).astype(np.float32)
        hidden = to_bf16_bits(h) if bf16 else h
    else:
        hidden = _values(rng, (B, Lh, wl.H), wl.value_std, bf16)
    q = _values(rng, (B, Lb, wl.Hq, wl.D), wl.value_std, bf16)
    k_blk = _values(rng, (B, Lb, wl.Hkv, wl.D), wl.value_std, bf16)
    v_blk = _values(rng, (B, Lb, wl.Hkv, wl.D), wl.value_std, bf16)
    C = wl.capacity
    if with_cache:
        k_cache = _values(rng, (B, wl.Hkv, C, wl.D), wl.value_std, bf16)
        v_cache = _values(rng, (B, wl.Hkv, C, wl.D), wl.value_std, bf16)
    else:
        k_cache = np.zeros((B, wl.Hkv, 0, wl.D), dtype=np.uint16 if bf16 else np.float32)
        v_cache = k_cache
    lo, hi = wl.ctx
    ctx_lens = rng.integers(lo, hi + 1, size=B, dtype=np.int64).astype(np.int32)
    prompt_ids = rng.integers(0, wl.V, size=wl.n_prompt, dtype=np.int64).astype(np.int32)
    prefix_ids = rng.integers(0, wl.V, size=(B, wl.n_prefix_eff), dtype=np.int64).astype(np.int32)
    draft_keep = rng.random((B, wl.gamma)) < wl.p_argmax
    if wl.draft_dist == "uniform":
        draft_alt = rng.integers(0, wl.V, size=(B, wl.gamma), dtype=np.int64).astype(np.int32)
    elif wl.draft_dist == "zipf1.1":
        draft_alt = _zipf_ids(rng, B * wl.gamma, wl.V).reshape(B, wl.gamma)
    else:
        raise ValueError(wl.draft_dist)
    return VerifyInputs(wl, W, hidden, q, k_blk, v_blk, k_cache, v_cache, ctx_lens,
                        prompt_ids, prefix_ids, draft_keep, draft_alt)


def make_drafts(inp: VerifyInputs, target_choice: np.ndarray) -> np.ndarray:
    """Drafts = target's choice where ``draft_keep`` else ``draft_alt``.

    ``target_choice`` is [B, gamma] (the target's argmax at each draft
    position); the caller computes it.
    """
    tc = np.asarray(target_choice, dtype=np.int32).reshape(inp.wl.B, inp.wl.gamma)
    return np.where(inp.draft_keep, tc, inp.draft_alt).astype(np.int32)
