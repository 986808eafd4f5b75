"""Thin ctypes binding of ``librv.so`` (declared in ``include/rv.h``).

Argument marshalling only: every function passes tensor data pointers, sizes
and the CUDA stream to the C entry point of the same name and raises
``RVError`` on a negative status.  All compute happens in the library's CUDA
kernels.  Importing this module fails loudly (``RVLibraryMissing``) when the
library has not been built; there is no other code path.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "librv.so")

RV_OK = 0
RV_ERR_INVALID_ARG = -1
RV_ERR_SHAPE = -2
RV_ERR_CAPACITY = -3
RV_ERR_CUDA = -4
RV_ERR_NOT_IMPLEMENTED = -5
RV_ERR_UNSUPPORTED = -6
RV_ERR_DEVICE = -7

RV_DEV_CTX_RANGE = 1
RV_DEV_DRAFT_RANGE = 2
RV_DEV_TIMEOUT = 4

RV_DTYPE_BF16 = 0
RV_DTYPE_F32 = 1

RV_NSCORES = 7
RV_SCORE_LSE_ORIG, RV_SCORE_LSE_REFL, RV_SCORE_LSE_FUSED = 0, 1, 2
RV_SCORE_LOGP_FUSED, RV_SCORE_LOGP_ORIG, RV_SCORE_LOGP_REFL = 3, 4, 5
RV_SCORE_ENT_ORIG = 6

RV_ACCEPT_EXACT, RV_ACCEPT_TYPICAL, RV_ACCEPT_SPECULATIVE, RV_ACCEPT_SAMPLED = 0, 1, 2, 3
RV_ACCEPT_TYPICAL_SAMPLED = 4
RV_HEAD_FUSED_LOGITS, RV_HEAD_PREBLENDED, RV_HEAD_STANDARD = 0, 1, 2

RV_PROF_ATTENTION, RV_PROF_HEAD_GEMM, RV_PROF_HEAD, RV_PROF_ACCEPT = 0, 1, 2, 3
RV_PROF_COUNT = 4


class RVLibraryMissing(ImportError):
    pass


class RVError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"rv error {code}: {msg}")
        self.code = code


class rv_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "hidden", "vocab", "n_q_heads", "n_kv_heads", "head_dim", "max_batch", "max_gamma",
        "max_template", "max_ctx", "dtype")]


def _load():
    if not os.path.exists(LIB_PATH):
        raise RVLibraryMissing(
            f"{LIB_PATH} is missing: build it with `python -m paper_2505_18629_gb300.build`")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, F, U64P = ctypes.c_void_p, ctypes.c_int32, ctypes.c_float, ctypes.POINTER(ctypes.c_uint64)
    sig = {
        "rv_create": (I, [ctypes.POINTER(rv_config), ctypes.POINTER(P)]),
        "rv_destroy": (I, [P]),
        "rv_last_error": (ctypes.c_char_p, [P]),
        "rv_workspace_bytes": (I, [P, U64P]),
        "rv_pack_block": (I, [P, P, P, P, P, I, I, I, I, P, P, P]),
        "rv_pack_block_pending": (I, [P, P, P, P, P, P, I, I, I, I, P, P, P]),
        "rv_verify_step_pending": (I, [P, P, P, P, P, P, P, P, P, P, P, P, P, I, I, I, I, F, P, P, P,
                                       P, P, P, P, P, P, P, P]),
        "rv_verify_attention": (I, [P, P, P, P, P, P, P, I, I, P, P]),
        "rv_verify_head": (I, [P, P, P, P, I, I, I, F, P, P, P, P]),
        "rv_accept": (I, [P, P, P, I, I, P, P, P, P, P, P]),
        "rv_accept_typical": (I, [P, P, P, P, I, I, F, F, P, P, P, P, P, P]),
        "rv_set_acceptance": (I, [P, I, F, F]),
        "rv_set_head_mode": (I, [P, I]),
        "rv_host_step_graphed": (I, [P, P]),
        "rv_accept_speculative": (I, [P, P, P, P, P, P, I, I, P, P, P, P, P, P]),
        "rv_verify_step_speculative": (I, [P, P, P, P, P, P, P, P, P, P, P, P, I, I, I, I, F, P, P,
                                           P, P, P, P, P, P, P, P, P, P, P, P]),
        "rv_accept_sampled": (I, [P, P, P, F, I, I, P, P, P, P, P, P, P]),
        "rv_verify_step_sampled": (I, [P, P, P, P, P, P, P, P, P, P, P, P, I, I, I, I, F, F, P, P,
                                       P, P, P, P, P, P, P, P, P, P, P]),
        "rv_verify_step": (I, [P, P, P, P, P, P, P, P, P, P, P, P, I, I, I, I, F, P, P, P, P, P, P,
                               P, P, P, P, P]),
        "rv_verify_step_host": (I, [P, P, P, P, P, P, P, P, P, P, P, P, I, I, I, I, F, P, P, P, P,
                                    P, P, P, P, P, P, U64P, U64P, P]),
        "rv_verify_head_static": (I, [P, P, P, I, I, I, I, I, F, P, P, P, P, P]),
        "rv_read_status": (I, [P, P, ctypes.POINTER(ctypes.c_uint32)]),
        "rv_profile_enable": (I, [P, I]),
        "rv_profile_read": (I, [P, I, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(I)]),
        "rv_launch_count": (I, [P, U64P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = _load()


def lib():
    return _lib


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, torch.Tensor):
        if not t.is_contiguous():
            raise ValueError("tensor arguments must be contiguous")
        return ctypes.c_void_p(t.data_ptr())
    return t


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


# ------------------------------------------------------------------ argument checks
# The C entry points take bare pointers, so they cannot see a tensor's size: a
# hidden-state tensor with too few rows would be read past its end on the
# device.  Every wrapper therefore checks shapes and element types against the
# sizes it passes (and the handle's configuration) and raises ValueError before
# anything is launched.

def _expect(name, t, shape, dtype, device=True, min_first=False):
    """One tensor: shape (first dimension at least shape[0] with min_first),
    dtype, contiguity and, unless device is None, device (True) or host
    (False) memory."""
    if t is None:
        raise ValueError(f"{name} is required")
    if not isinstance(t, torch.Tensor):
        raise ValueError(f"{name} must be a torch.Tensor")
    got = tuple(t.shape)
    want = tuple(int(x) for x in shape)
    if min_first:
        ok = len(got) == len(want) and got[0] >= want[0] and got[1:] == want[1:]
    else:
        ok = got == want
    if not ok:
        lead = ">= " if min_first else ""
        raise ValueError(f"{name} has shape {list(got)}, expected {lead}{list(want)}")
    if t.dtype != dtype:
        raise ValueError(f"{name} has dtype {t.dtype}, expected {dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if device is not None and t.is_cuda != device:
        raise ValueError(f"{name} must be in {'device' if device else 'host'} memory")


class _Checks:
    """Shapes and dtypes of every tensor first, then where each one lives, so
    that a wrong shape is reported as such whatever the memory."""

    def __init__(self):
        self._where = []

    def __call__(self, name, t, shape, dtype, device=True, min_first=False):
        _expect(name, t, shape, dtype, None, min_first)
        self._where.append((name, t, device))

    def placed(self):
        for name, t, device in self._where:
            if device is not None and t.is_cuda != device:
                raise ValueError(f"{name} must be in {'device' if device else 'host'} memory")


def _block_len(h, gamma, R):
    """Block positions without the pending token: [x, template, x], or the
    drafts alone for standard verification."""
    return gamma if h.head_mode == RV_HEAD_STANDARD else 2 * gamma + R


def _check_head(h, hidden, w_head, draft_ids, gamma, R, scores, argmax, margin, device=True,
                ck=None):
    own = ck is None
    ck = _Checks() if own else ck
    c = h.cfg
    act = h.act_dtype
    if hidden is None or hidden.dim() != 3:
        raise ValueError("hidden must be [B, Lb + 1, H]")
    B = hidden.shape[0]
    ck("hidden", hidden, (B, _block_len(h, gamma, R) + 1, c.hidden), act, device)
    ck("w_head", w_head, (c.vocab, c.hidden), act, True)
    ck("draft_ids", draft_ids, (B, gamma), torch.int32, device)
    ck("scores", scores, (B, gamma + 1, RV_NSCORES), torch.float32, device)
    ck("argmax", argmax, (B, gamma + 1), torch.int32, device)
    ck("margin", margin, (B, gamma), torch.float32, device)
    if own:
        ck.placed()
    return B


def _check_attention(h, q, k_blk, v_blk, k_cache, v_cache, ctx_lens, out, B, Lq, device=True,
                     ck=None):
    own = ck is None
    ck = _Checks() if own else ck
    c = h.cfg
    act = h.act_dtype
    ck("q", q, (B, Lq, c.n_q_heads, c.head_dim), act, device)
    ck("k_blk", k_blk, (B, Lq, c.n_kv_heads, c.head_dim), act, device)
    ck("v_blk", v_blk, (B, Lq, c.n_kv_heads, c.head_dim), act, device)
    ck("k_cache", k_cache, (B, c.n_kv_heads, c.max_ctx, c.head_dim), act, True, min_first=True)
    ck("v_cache", v_cache, (B, c.n_kv_heads, c.max_ctx, c.head_dim), act, True, min_first=True)
    ck("ctx_lens", ctx_lens, (B,), torch.int32, device)
    if out is not None:
        ck("attn_out", out, (B, Lq, c.n_q_heads, c.head_dim), act, device)
    if own:
        ck.placed()


def _check_ids(B, gamma, draft_ids, prompt_ids, prefix_ids, device=True, ck=None):
    own = ck is None
    ck = _Checks() if own else ck
    ck("draft_ids", draft_ids, (B, gamma), torch.int32, device)
    if prompt_ids is not None:
        ck("prompt_ids", prompt_ids, (prompt_ids.numel(),), torch.int32, device)
    if prefix_ids is None or prefix_ids.dim() != 2:
        raise ValueError("prefix_ids must be [B, n_prefix]")
    ck("prefix_ids", prefix_ids, (B, prefix_ids.shape[1]), torch.int32, device)
    if own:
        ck.placed()


def _check_accept_out(B, gamma, accept_mask, accepted_len, next_token, ctx_in, ctx_out,
                      device=True, ck=None):
    own = ck is None
    ck = _Checks() if own else ck
    ck("accept_mask", accept_mask, (B, gamma), torch.uint8, device)
    ck("accepted_len", accepted_len, (B,), torch.int32, device)
    ck("next_token", next_token, (B,), torch.int32, device)
    ck("ctx_in", ctx_in, (B,), torch.int32, device)
    ck("ctx_out", ctx_out, (B,), torch.int32, device)
    if own:
        ck.placed()


def _check_step(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                accept_mask, accepted_len, next_token, ctx_out, lead=0, device=True):
    """Shapes of a whole step; lead = 1 for the pending-token block."""
    if draft_ids is None or draft_ids.dim() != 2:
        raise ValueError("draft_ids must be [B, gamma]")
    ck = _Checks()
    B, gamma = draft_ids.shape
    _check_ids(B, gamma, draft_ids, prompt_ids, prefix_ids, device, ck)
    n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
    R = n_prompt + prefix_ids.shape[1]
    Lq = _block_len(h, gamma, R) + lead
    _check_attention(h, q, k_blk, v_blk, k_cache, v_cache, ctx_in, attn_out, B, Lq, device, ck)
    _check_head(h, hidden, w_head, draft_ids, gamma, R, scores, argmax, margin, device, ck)
    if block_ids is not None or pos_ids is not None:
        ck("block_ids", block_ids, (B, Lq), torch.int32, device)
        ck("pos_ids", pos_ids, (B, Lq), torch.int32, device)
    _check_accept_out(B, gamma, accept_mask, accepted_len, next_token, ctx_in, ctx_out, device, ck)
    ck.placed()


def _check_speculative_inputs(h, B, gamma, q_draft, r_uniform, u_uniform):
    _expect("q_draft", q_draft, (B, gamma, h.cfg.vocab), torch.float32)
    _expect("r_uniform", r_uniform, (B, gamma), torch.float32)
    _expect("u_uniform", u_uniform, (B,), torch.float32)


def _check_sampled_inputs(B, gamma, u_uniform, sampled):
    _expect("u_uniform", u_uniform, (B, gamma + 1), torch.float32)
    _expect("sampled", sampled, (B, gamma + 1), torch.int32)


class Handle:
    """Owns an ``rv_handle*``; ``close()`` (or garbage collection) destroys it."""

    def __init__(self, ptr, cfg):
        self._p = ptr
        self.cfg = cfg
        self.head_mode = RV_HEAD_FUSED_LOGITS  # last mode set by rv_set_head_mode

    @property
    def act_dtype(self):
        """Element type of hidden states, weight, q/k/v and caches."""
        return torch.bfloat16 if self.cfg.dtype == RV_DTYPE_BF16 else torch.float32

    @property
    def ptr(self):
        if not self._p:
            raise ValueError("handle is closed")
        return self._p

    def close(self):
        if self._p:
            _lib.rv_destroy(self._p)
            self._p = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def last_error(self) -> str:
        return _lib.rv_last_error(self._p).decode()


def _check(h, rc):
    if rc != RV_OK:
        msg = _lib.rv_last_error(h.ptr if isinstance(h, Handle) else h)
        raise RVError(rc, msg.decode() if msg else "")
    return rc


def rv_create(hidden, vocab, n_q_heads, n_kv_heads, head_dim, max_batch, max_gamma,
              max_template, max_ctx, dtype=RV_DTYPE_BF16) -> Handle:
    cfg = rv_config(hidden, vocab, n_q_heads, n_kv_heads, head_dim, max_batch, max_gamma,
                    max_template, max_ctx, dtype)
    out = ctypes.c_void_p()
    rc = _lib.rv_create(ctypes.byref(cfg), ctypes.byref(out))
    if rc != RV_OK:
        raise RVError(rc, _lib.rv_last_error(None).decode())
    return Handle(out, cfg)


def rv_workspace_bytes(h: Handle) -> int:
    v = ctypes.c_uint64()
    _check(h, _lib.rv_workspace_bytes(h.ptr, ctypes.byref(v)))
    return v.value


def rv_pack_block(h, draft_ids, prompt_ids, prefix_ids, ctx_lens, block_ids, pos_ids,
                  stream=None):
    B, gamma = draft_ids.shape
    _check_ids(B, gamma, draft_ids, prompt_ids, prefix_ids)
    n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
    n_prefix = prefix_ids.shape[1]
    Lb = _block_len(h, gamma, n_prompt + n_prefix)
    _expect("ctx_lens", ctx_lens, (B,), torch.int32)
    _expect("block_ids", block_ids, (B, Lb), torch.int32)
    _expect("pos_ids", pos_ids, (B, Lb), torch.int32)
    _check(h, _lib.rv_pack_block(h.ptr, _ptr(draft_ids), _ptr(prompt_ids), _ptr(prefix_ids),
                                 _ptr(ctx_lens), B, gamma, n_prompt, n_prefix, _ptr(block_ids),
                                 _ptr(pos_ids), _stream(stream)))


def rv_pack_block_pending(h, pending_ids, draft_ids, prompt_ids, prefix_ids, ctx_lens, block_ids,
                          pos_ids, stream=None):
    B, gamma = draft_ids.shape
    _check_ids(B, gamma, draft_ids, prompt_ids, prefix_ids)
    n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
    n_prefix = prefix_ids.shape[1]
    Lb = _block_len(h, gamma, n_prompt + n_prefix)
    _expect("pending_ids", pending_ids, (B,), torch.int32)
    _expect("ctx_lens", ctx_lens, (B,), torch.int32)
    _expect("block_ids", block_ids, (B, Lb + 1), torch.int32)
    _expect("pos_ids", pos_ids, (B, Lb + 1), torch.int32)
    _check(h, _lib.rv_pack_block_pending(h.ptr, _ptr(pending_ids), _ptr(draft_ids),
                                         _ptr(prompt_ids), _ptr(prefix_ids), _ptr(ctx_lens), B,
                                         gamma, n_prompt, n_prefix, _ptr(block_ids), _ptr(pos_ids),
                                         _stream(stream)))


def rv_verify_attention(h, q, k_blk, v_blk, k_cache, v_cache, ctx_lens, out, stream=None):
    if q is None or q.dim() != 4:
        raise ValueError("q must be [B, Lb, Hq, D]")
    B, Lb = q.shape[0], q.shape[1]
    _check_attention(h, q, k_blk, v_blk, k_cache, v_cache, ctx_lens, out, B, Lb)
    if out is None:
        raise ValueError("out is required")
    _check(h, _lib.rv_verify_attention(h.ptr, _ptr(q), _ptr(k_blk), _ptr(v_blk), _ptr(k_cache),
                                       _ptr(v_cache), _ptr(ctx_lens), B, Lb, _ptr(out),
                                       _stream(stream)))


def rv_verify_head(h, hidden, w_head, draft_ids, gamma, R, alpha, scores, argmax, margin,
                   stream=None):
    B = _check_head(h, hidden, w_head, draft_ids, gamma, R, scores, argmax, margin)
    _check(h, _lib.rv_verify_head(h.ptr, _ptr(hidden), _ptr(w_head), _ptr(draft_ids), B, gamma,
                                  R, float(alpha), _ptr(scores), _ptr(argmax), _ptr(margin),
                                  _stream(stream)))


def rv_accept(h, draft_ids, argmax, accept_mask, accepted_len, next_token, ctx_in, ctx_out,
              stream=None):
    B, gamma = draft_ids.shape
    _expect("draft_ids", draft_ids, (B, gamma), torch.int32)
    _expect("argmax", argmax, (B, gamma + 1), torch.int32)
    _check_accept_out(B, gamma, accept_mask, accepted_len, next_token, ctx_in, ctx_out)
    _check(h, _lib.rv_accept(h.ptr, _ptr(draft_ids), _ptr(argmax), B, gamma, _ptr(accept_mask),
                             _ptr(accepted_len), _ptr(next_token), _ptr(ctx_in), _ptr(ctx_out),
                             _stream(stream)))


def rv_accept_typical(h, draft_ids, scores, argmax, eps, delta, accept_mask, accepted_len,
                      next_token, ctx_in, ctx_out, stream=None):
    B, gamma = draft_ids.shape
    _expect("draft_ids", draft_ids, (B, gamma), torch.int32)
    _expect("scores", scores, (B, gamma + 1, RV_NSCORES), torch.float32)
    _expect("argmax", argmax, (B, gamma + 1), torch.int32)
    _check_accept_out(B, gamma, accept_mask, accepted_len, next_token, ctx_in, ctx_out)
    _check(h, _lib.rv_accept_typical(h.ptr, _ptr(draft_ids), _ptr(scores), _ptr(argmax), B, gamma,
                                     float(eps), float(delta), _ptr(accept_mask),
                                     _ptr(accepted_len), _ptr(next_token), _ptr(ctx_in),
                                     _ptr(ctx_out), _stream(stream)))


def rv_accept_speculative(h, draft_ids, q_draft, r_uniform, u_uniform, scores, accept_mask,
                          accepted_len, next_token, ctx_in, ctx_out, stream=None):
    B, gamma = draft_ids.shape
    _expect("draft_ids", draft_ids, (B, gamma), torch.int32)
    _check_speculative_inputs(h, B, gamma, q_draft, r_uniform, u_uniform)
    _expect("scores", scores, (B, gamma + 1, RV_NSCORES), torch.float32)
    _check_accept_out(B, gamma, accept_mask, accepted_len, next_token, ctx_in, ctx_out)
    _check(h, _lib.rv_accept_speculative(h.ptr, _ptr(draft_ids), _ptr(q_draft), _ptr(r_uniform),
                                         _ptr(u_uniform), _ptr(scores), B, gamma, _ptr(accept_mask),
                                         _ptr(accepted_len), _ptr(next_token), _ptr(ctx_in),
                                         _ptr(ctx_out), _stream(stream)))


def rv_accept_sampled(h, draft_ids, u_uniform, temperature, sampled, accept_mask, accepted_len,
                      next_token, ctx_in, ctx_out, stream=None):
    B, gamma = draft_ids.shape
    _expect("draft_ids", draft_ids, (B, gamma), torch.int32)
    _check_sampled_inputs(B, gamma, u_uniform, sampled)
    _check_accept_out(B, gamma, accept_mask, accepted_len, next_token, ctx_in, ctx_out)
    _check(h, _lib.rv_accept_sampled(h.ptr, _ptr(draft_ids), _ptr(u_uniform), float(temperature),
                                     B, gamma, _ptr(sampled), _ptr(accept_mask),
                                     _ptr(accepted_len), _ptr(next_token), _ptr(ctx_in),
                                     _ptr(ctx_out), _stream(stream)))


def rv_host_step_graphed(h):
    """True when the handle replays a CUDA graph for its repeated host-buffer step."""
    v = ctypes.c_int32()
    _check(h, _lib.rv_host_step_graphed(h.ptr, ctypes.byref(v)))
    return bool(v.value)


def rv_set_head_mode(h, mode):
    _check(h, _lib.rv_set_head_mode(h.ptr, int(mode)))
    h.head_mode = int(mode)


def rv_set_acceptance(h, mode, eps=0.0, delta=0.0):
    _check(h, _lib.rv_set_acceptance(h.ptr, int(mode), float(eps), float(delta)))


def rv_verify_step(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                   prefix_ids, ctx_in, alpha, block_ids, pos_ids, attn_out, scores, argmax, margin,
                   accept_mask, accepted_len, next_token, ctx_out, stream=None):
    """Whole step; prompt_ids may be None (empty prompt), block_ids None skips packing."""
    _check_step(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                accept_mask, accepted_len, next_token, ctx_out)
    B, gamma = draft_ids.shape
    n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
    n_prefix = prefix_ids.shape[1]
    _check(h, _lib.rv_verify_step(
        h.ptr, _ptr(q), _ptr(k_blk), _ptr(v_blk), _ptr(k_cache), _ptr(v_cache), _ptr(hidden),
        _ptr(w_head), _ptr(draft_ids), _ptr(prompt_ids), _ptr(prefix_ids), _ptr(ctx_in), B, gamma,
        n_prompt, n_prefix, float(alpha), _ptr(block_ids), _ptr(pos_ids), _ptr(attn_out),
        _ptr(scores), _ptr(argmax), _ptr(margin), _ptr(accept_mask), _ptr(accepted_len),
        _ptr(next_token), _ptr(ctx_out), _stream(stream)))


def rv_verify_step_pending(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, pending_ids,
                           draft_ids, prompt_ids, prefix_ids, ctx_in, alpha, block_ids, pos_ids,
                           attn_out, scores, argmax, margin, accept_mask, accepted_len, next_token,
                           ctx_out, stream=None):
    """Whole step over the pending-token block [t, x, template, x] (Lb + 1 positions)."""
    _check_step(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                accept_mask, accepted_len, next_token, ctx_out, lead=1)
    B, gamma = draft_ids.shape
    _expect("pending_ids", pending_ids, (B,), torch.int32)
    n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
    n_prefix = prefix_ids.shape[1]
    _check(h, _lib.rv_verify_step_pending(
        h.ptr, _ptr(q), _ptr(k_blk), _ptr(v_blk), _ptr(k_cache), _ptr(v_cache), _ptr(hidden),
        _ptr(w_head), _ptr(pending_ids), _ptr(draft_ids), _ptr(prompt_ids), _ptr(prefix_ids),
        _ptr(ctx_in), B, gamma, n_prompt, n_prefix, float(alpha), _ptr(block_ids), _ptr(pos_ids),
        _ptr(attn_out), _ptr(scores), _ptr(argmax), _ptr(margin), _ptr(accept_mask),
        _ptr(accepted_len), _ptr(next_token), _ptr(ctx_out), _stream(stream)))


def rv_verify_step_speculative(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids,
                               prompt_ids, prefix_ids, ctx_in, alpha, q_draft, r_uniform,
                               u_uniform, block_ids, pos_ids, attn_out, scores, argmax, margin,
                               accept_mask, accepted_len, next_token, ctx_out, stream=None):
    """Whole step with the speculative-sampling acceptance (Alg. 1)."""
    _check_step(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                accept_mask, accepted_len, next_token, ctx_out)
    B, gamma = draft_ids.shape
    _check_speculative_inputs(h, B, gamma, q_draft, r_uniform, u_uniform)
    n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
    n_prefix = prefix_ids.shape[1]
    _check(h, _lib.rv_verify_step_speculative(
        h.ptr, _ptr(q), _ptr(k_blk), _ptr(v_blk), _ptr(k_cache), _ptr(v_cache), _ptr(hidden),
        _ptr(w_head), _ptr(draft_ids), _ptr(prompt_ids), _ptr(prefix_ids), _ptr(ctx_in), B, gamma,
        n_prompt, n_prefix, float(alpha), _ptr(q_draft), _ptr(r_uniform), _ptr(u_uniform),
        _ptr(block_ids), _ptr(pos_ids), _ptr(attn_out), _ptr(scores), _ptr(argmax), _ptr(margin),
        _ptr(accept_mask), _ptr(accepted_len), _ptr(next_token), _ptr(ctx_out), _stream(stream)))


def rv_verify_step_sampled(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids,
                           prompt_ids, prefix_ids, ctx_in, alpha, temperature, u_uniform,
                           block_ids, pos_ids, attn_out, scores, argmax, margin, sampled,
                           accept_mask, accepted_len, next_token, ctx_out, stream=None):
    """Whole step with exact match against target tokens sampled at temperature T (Alg. 2)."""
    _check_step(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                accept_mask, accepted_len, next_token, ctx_out)
    B, gamma = draft_ids.shape
    _check_sampled_inputs(B, gamma, u_uniform, sampled)
    n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
    n_prefix = prefix_ids.shape[1]
    _check(h, _lib.rv_verify_step_sampled(
        h.ptr, _ptr(q), _ptr(k_blk), _ptr(v_blk), _ptr(k_cache), _ptr(v_cache), _ptr(hidden),
        _ptr(w_head), _ptr(draft_ids), _ptr(prompt_ids), _ptr(prefix_ids), _ptr(ctx_in), B, gamma,
        n_prompt, n_prefix, float(alpha), float(temperature), _ptr(u_uniform), _ptr(block_ids),
        _ptr(pos_ids), _ptr(attn_out), _ptr(scores), _ptr(argmax), _ptr(margin), _ptr(sampled),
        _ptr(accept_mask), _ptr(accepted_len), _ptr(next_token), _ptr(ctx_out), _stream(stream)))


def rv_verify_step_host(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids,
                        prompt_ids, prefix_ids, ctx_in, alpha, block_ids, pos_ids, attn_out,
                        scores, argmax, margin, accept_mask, accepted_len, next_token, ctx_out,
                        stream=None):
    """Host tensors in/out (pin them for asynchronous copies); returns (h2d, d2h) bytes."""
    _check_step(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                accept_mask, accepted_len, next_token, ctx_out, device=False)
    B, gamma = draft_ids.shape
    n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
    n_prefix = prefix_ids.shape[1]
    hb, db = ctypes.c_uint64(), ctypes.c_uint64()
    _check(h, _lib.rv_verify_step_host(
        h.ptr, _ptr(q), _ptr(k_blk), _ptr(v_blk), _ptr(k_cache), _ptr(v_cache), _ptr(hidden),
        _ptr(w_head), _ptr(draft_ids), _ptr(prompt_ids), _ptr(prefix_ids), _ptr(ctx_in), B, gamma,
        n_prompt, n_prefix, float(alpha), _ptr(block_ids), _ptr(pos_ids), _ptr(attn_out),
        _ptr(scores), _ptr(argmax), _ptr(margin), _ptr(accept_mask), _ptr(accepted_len),
        _ptr(next_token), _ptr(ctx_out), ctypes.byref(hb), ctypes.byref(db), _stream(stream)))
    return hb.value, db.value


class PreparedStep:
    """rv_verify_step with its arguments checked and marshalled once.

    For loops that run the same step on the same device buffers (a serving
    loop's persistent inputs and outputs, a benchmark): the shape checks and
    ~30 ctypes arguments cost tens of microseconds of Python per call, which
    this pays once.  Calling the object runs the same C entry point."""

    def __init__(self, h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids,
                 prompt_ids, prefix_ids, ctx_in, alpha, block_ids, pos_ids, attn_out, scores,
                 argmax, margin, accept_mask, accepted_len, next_token, ctx_out, stream=None):
        _check_step(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                    prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                    accept_mask, accepted_len, next_token, ctx_out)
        B, gamma = draft_ids.shape
        n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
        n_prefix = prefix_ids.shape[1]
        self._h = h
        self._keep = (q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                      prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                      accept_mask, accepted_len, next_token, ctx_out)
        self._fn = _lib.rv_verify_step
        self._args = (
            h.ptr, _ptr(q), _ptr(k_blk), _ptr(v_blk), _ptr(k_cache), _ptr(v_cache), _ptr(hidden),
            _ptr(w_head), _ptr(draft_ids), _ptr(prompt_ids), _ptr(prefix_ids), _ptr(ctx_in), B,
            gamma, n_prompt, n_prefix, float(alpha), _ptr(block_ids), _ptr(pos_ids),
            _ptr(attn_out), _ptr(scores), _ptr(argmax), _ptr(margin), _ptr(accept_mask),
            _ptr(accepted_len), _ptr(next_token), _ptr(ctx_out), _stream(stream))

    def __call__(self):
        rc = self._fn(*self._args)
        if rc != RV_OK:
            _check(self._h, rc)


class PreparedStepHost:
    """rv_verify_step_host with its arguments marshalled once.

    For loops that reuse the same host and device buffers every step (a serving
    loop's pinned staging): building ~30 ctypes arguments costs tens of
    microseconds of Python per call, which this pays once.  Calling the object
    runs the same C entry point; it returns (h2d, d2h) bytes of the step."""

    def __init__(self, h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids,
                 prompt_ids, prefix_ids, ctx_in, alpha, block_ids, pos_ids, attn_out, scores,
                 argmax, margin, accept_mask, accepted_len, next_token, ctx_out, stream=None):
        _check_step(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                    prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                    accept_mask, accepted_len, next_token, ctx_out, device=False)
        B, gamma = draft_ids.shape
        n_prompt = 0 if prompt_ids is None else prompt_ids.numel()
        n_prefix = prefix_ids.shape[1]
        self._h = h
        self._keep = (q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                      prefix_ids, ctx_in, block_ids, pos_ids, attn_out, scores, argmax, margin,
                      accept_mask, accepted_len, next_token, ctx_out)
        self._hb, self._db = ctypes.c_uint64(), ctypes.c_uint64()
        self._fn = _lib.rv_verify_step_host
        self._args = (
            h.ptr, _ptr(q), _ptr(k_blk), _ptr(v_blk), _ptr(k_cache), _ptr(v_cache), _ptr(hidden),
            _ptr(w_head), _ptr(draft_ids), _ptr(prompt_ids), _ptr(prefix_ids), _ptr(ctx_in), B,
            gamma, n_prompt, n_prefix, float(alpha), _ptr(block_ids), _ptr(pos_ids),
            _ptr(attn_out), _ptr(scores), _ptr(argmax), _ptr(margin), _ptr(accept_mask),
            _ptr(accepted_len), _ptr(next_token), _ptr(ctx_out), ctypes.byref(self._hb),
            ctypes.byref(self._db), _stream(stream))

    def __call__(self):
        rc = self._fn(*self._args)
        if rc != RV_OK:
            _check(self._h, rc)
        return self._hb.value, self._db.value


RV_STATIC_MAX_PAIRS = 64
RV_STATIC_MAX_HIDDEN = 8192


def rv_verify_head_static(hidden, w_head, draft_ids, gamma, R, alpha, scores, argmax, margin,
                          dev_status=None, stream=None):
    """rv_verify_head without a handle or any device allocation (fixed internal
    scratch; limits RV_STATIC_MAX_PAIRS / RV_STATIC_MAX_HIDDEN)."""
    if hidden is None or hidden.dim() != 3 or w_head is None or w_head.dim() != 2:
        raise ValueError("hidden must be [B, 2*gamma+R+1, H] and w_head [V, H]")
    B = hidden.shape[0]
    V, H = w_head.shape
    ck = _Checks()
    ck("hidden", hidden, (B, 2 * gamma + R + 1, H), torch.bfloat16)
    ck("w_head", w_head, (V, H), torch.bfloat16)
    ck("draft_ids", draft_ids, (B, gamma), torch.int32)
    ck("scores", scores, (B, gamma + 1, RV_NSCORES), torch.float32)
    ck("argmax", argmax, (B, gamma + 1), torch.int32)
    ck("margin", margin, (B, gamma), torch.float32)
    if dev_status is not None:
        ck("dev_status", dev_status, (1,), torch.int32)
    ck.placed()
    rc = _lib.rv_verify_head_static(_ptr(hidden), _ptr(w_head), _ptr(draft_ids), B, gamma, R, V,
                                    H, float(alpha), _ptr(scores), _ptr(argmax), _ptr(margin),
                                    _ptr(dev_status), _stream(stream))
    if rc != RV_OK:
        raise RVError(rc, "rv_verify_head_static")


def rv_read_status(h, stream=None) -> int:
    """Synchronizes; returns the device status bits (and clears them)."""
    st = ctypes.c_uint32()
    rc = _lib.rv_read_status(h.ptr, _stream(stream), ctypes.byref(st))
    if rc not in (RV_OK, RV_ERR_DEVICE):
        _check(h, rc)
    return st.value


def rv_profile_enable(h, mask):
    """mask: bit (1 << RV_PROF_*) per region to record; 0 stops."""
    _check(h, _lib.rv_profile_enable(h.ptr, int(mask)))


def rv_profile_read(h, region):
    ms, n = ctypes.c_double(), ctypes.c_int32()
    _check(h, _lib.rv_profile_read(h.ptr, region, ctypes.byref(ms), ctypes.byref(n)))
    return ms.value, n.value


def rv_launch_count(h) -> int:
    v = ctypes.c_uint64()
    _check(h, _lib.rv_launch_count(h.ptr, ctypes.byref(v)))
    return v.value
