"""Python binding of libcospec.so: the calls of include/cospec.h, same names.

Argument marshalling only -- shapes are read off the tensors and checked
against one another (a mis-shaped tensor would make a kernel read or write
past its end), pointers and the current CUDA stream are passed through
ctypes, and every step runs in the library's CUDA kernels.  There is no CPU or PyTorch fallback: if the
library is missing or a call fails, an exception is raised.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libcospec.so")

POLICY_MLP, POLICY_TARGET, POLICY_DRAFT = 0, 1, 2
DEVERR_PAGE, DEVERR_CTX, DEVERR_TOKEN, DEVERR_TIMEOUT, DEVERR_OFFSETS = 1, 2, 4, 8, 16

EXPORTED = ("cospec_status_string", "cospec_last_cuda_error", "cospec_get_device_error", "cospec_num_sms",
            "cospec_verify_attn", "cospec_lmhead_workspace", "cospec_lmhead_argmax_features",
            "cospec_arbitrate", "cospec_accept_commit", "cospec_lmhead_argmax_features_noalloc",
            "cospec_lmhead_sample_features", "cospec_verify_attn_plan", "cospec_rl_workspace",
            "cospec_rl_advantages", "cospec_verify_attn_plan_model",
            "cospec_lmhead_logits_features", "cospec_sps_workspace", "cospec_sps_accept")


class AttnDims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int), ("rows", ctypes.c_int), ("num_q_heads", ctypes.c_int),
                ("num_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int),
                ("page_size", ctypes.c_int), ("max_pages_per_seq", ctypes.c_int),
                ("num_pages", ctypes.c_int), ("softmax_scale", ctypes.c_float),
                ("flags", ctypes.c_int)]


class RLParams(ctypes.Structure):
    """cospec_rl_params; defaults are the paper's (App. C)."""
    _fields_ = [(n, ctypes.c_float) for n in
                ("alpha", "beta", "eta_fail", "eps", "clip_eps", "beta_h", "beta_kl")]

    def __init__(self, alpha=1.0, beta=0.25, eta_fail=0.5, eps=1e-6, clip_eps=0.2, beta_h=0.01,
                 beta_kl=0.02):
        super().__init__(alpha, beta, eta_fail, eps, clip_eps, beta_h, beta_kl)


ATTN_KV_STABLE = 1
ATTN_BLOCK_FULL = 2


class CospecError(RuntimeError):
    pass


_lib: Optional[ctypes.CDLL] = None

_vp, _i, _sz, _f = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float
_PDIMS = ctypes.POINTER(AttnDims)
# cospec_resident_fn: (kernel, rows, block_rows, splits, user) -> resident clusters
RESIDENT_FN = ctypes.CFUNCTYPE(ctypes.c_longlong, _i, _i, _i, _i, _vp)


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libcospec.so (built by ``paper_2605_24793_gb300.build``)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise CospecError(f"{path} is missing; build it with python -m paper_2605_24793_gb300.build")
    lib = ctypes.CDLL(path)
    sig = {
        "cospec_status_string": (ctypes.c_char_p, [_i]),
        "cospec_last_cuda_error": (ctypes.c_char_p, []),
        "cospec_get_device_error": (_i, [ctypes.POINTER(_i), _vp]),
        "cospec_num_sms": (_i, []),
        "cospec_verify_attn": (_i, [_PDIMS, _i, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
        "cospec_verify_attn_plan": (_i, [_PDIMS, _i, ctypes.POINTER(_i), ctypes.POINTER(_i)]),
        "cospec_verify_attn_plan_model": (_i, [_PDIMS, _i, _i, RESIDENT_FN, _vp,
                                               ctypes.POINTER(_i), ctypes.POINTER(_i)]),
        "cospec_rl_workspace": (_sz, [_i, _i]),
        "cospec_rl_advantages": (_i, [_i, _i, _i, _i, _vp, _vp, _vp, _vp, _vp, _vp,
                                      ctypes.POINTER(RLParams), _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                      _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
        "cospec_lmhead_workspace": (_sz, [_i, _i, _i]),
        "cospec_lmhead_argmax_features": (_i, [_i, _i, _i, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
        "cospec_lmhead_argmax_features_noalloc": (_i, [_i, _i, _i, _vp, _vp, _vp, _vp, _vp, _vp]),
        "cospec_lmhead_sample_features": (_i, [_i, _i, _i, _vp, _vp, _vp, _f, _vp, _vp, _vp, _vp,
                                               _sz, _vp]),
        "cospec_lmhead_logits_features": (_i, [_i, _i, _i, _vp, _vp, _vp, _f, _vp, _vp, _vp, _vp,
                                               _sz, _vp]),
        "cospec_sps_workspace": (_sz, [_i]),
        "cospec_sps_accept": (_i, [_i, _i, _i, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz,
                                   _vp]),
        "cospec_arbitrate": (_i, [_i, _i, _vp, _vp, _vp, _i, _vp, _vp, _vp, _f, _f, _i, _vp, _vp, _vp]),
        "cospec_accept_commit": (_i, [_i, _i, _i, _PDIMS, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                      ctypes.c_longlong, _vp, _vp, _vp, _vp, _vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(status: int) -> None:
    if status != 0:
        lib = load_library()
        msg = lib.cospec_status_string(status).decode()
        if status == -4:   # COSPEC_ERR_CUDA: name the runtime error behind it
            msg += f": {lib.cospec_last_cuda_error().decode()}"
        raise CospecError(f"cospec call failed: {msg} ({status})")


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _req(t: torch.Tensor, dtype, name: str, ndim: Optional[int] = None):
    if t.dtype != dtype:
        raise TypeError(f"{name}: expected {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name}: must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name}: must be contiguous")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name}: expected {ndim} dims, got {t.dim()}")


def _need(cond: bool, msg: str) -> None:
    if not cond:
        raise ValueError(msg)


def _same_device(*tensors: Optional[torch.Tensor]) -> None:
    """Every tensor on the current CUDA device (the library launches there)."""
    dev = torch.cuda.current_device()
    for t in tensors:
        if t is not None and t.device.index != dev:
            raise ValueError(f"tensor on {t.device}, but the current device is cuda:{dev}")


def check_attn_shapes(q, k_blk, v_blk, k_pages, v_pages, page_table, ctx_len, out) -> None:
    """Shapes of one verify-attention call agree: q / out [B,R,Hq,D], block
    K/V [B,R,Hkv,D], pools [num_pages,Hkv,P,D], page_table [B,max_pages],
    ctx_len [B]."""
    _need(q.dim() == 4, "q must be [B, R, Hq, D]")
    B, R, Hq, D = q.shape
    _need(k_pages.dim() == 4, "k_pages must be [num_pages, Hkv, P, D]")
    _need(tuple(v_pages.shape) == tuple(k_pages.shape), "v_pages must have k_pages' shape")
    Hkv = k_pages.shape[1]
    _need(k_pages.shape[3] == D, "k_pages head_dim differs from q's")
    _need(tuple(k_blk.shape) == (B, R, Hkv, D), "k_blk must be [B, R, Hkv, D]")
    _need(tuple(v_blk.shape) == (B, R, Hkv, D), "v_blk must be [B, R, Hkv, D]")
    _need(tuple(out.shape) == tuple(q.shape), "out must have q's shape")
    _need(page_table.dim() == 2 and page_table.shape[0] == B, "page_table must be [B, max_pages]")
    _need(ctx_len.dim() == 1 and ctx_len.shape[0] == B, "ctx_len must be [B]")


def check_arbitrate_shapes(draft, argmax, stats, w1, b1, w2, mode, p_out, accept) -> None:
    """draft [B,K]; argmax B*(K+1) ids; stats B*(K+1)*5; p_out / accept B*K;
    for the MLP policy w1 [H,8], b1 [H], w2 [H]."""
    _need(draft.dim() == 2, "draft must be [B, K]")
    B, K = draft.shape
    _need(argmax.numel() == B * (K + 1) and stats.numel() == B * (K + 1) * 5,
          "argmax / stats must hold K+1 rows per sequence")
    _need(p_out.numel() == B * K and accept.numel() == B * K, "p_out / accept must hold B*K values")
    if mode == POLICY_MLP:
        _need(w1.dim() == 2 and w1.shape[1] == 8, "w1 must be [H, 8]")
        H = w1.shape[0]
        _need(b1.numel() == H and w2.numel() == H, "b1 / w2 must hold H values")


def check_commit_shapes(draft, argmax, accept, k_blk, v_blk, k_pages, v_pages, page_table,
                        ctx_len, accept_len, emitted) -> None:
    """draft [B,K]; argmax B*(K+1); accept B*K; block K/V [L,B,K+1,Hkv,D];
    pools [L or 1,num_pages,Hkv,P,D]; page_table [B,max_pages]; ctx_len,
    accept_len [B]; emitted B*(K+1)."""
    _need(draft.dim() == 2, "draft must be [B, K]")
    B, K = draft.shape
    _need(argmax.numel() == B * (K + 1), "argmax must hold K+1 ids per sequence")
    _need(accept.numel() == B * K, "accept must hold B*K values")
    _need(k_blk.dim() == 5 and tuple(v_blk.shape) == tuple(k_blk.shape),
          "k_blk / v_blk must both be [L, B, K+1, Hkv, D]")
    L = k_blk.shape[0]
    _need(k_pages.dim() == 5 and tuple(v_pages.shape) == tuple(k_pages.shape),
          "k_pages / v_pages must both be [L, num_pages, Hkv, P, D]")
    _need(k_pages.shape[0] in (L, 1), "pools must hold every layer, or one shared by all")
    _need(tuple(k_blk.shape[1:]) == (B, K + 1, k_pages.shape[2], k_pages.shape[4]),
          "k_blk must be [L, B, K+1, Hkv, D] with the pools' Hkv and D")
    _need(page_table.dim() == 2 and page_table.shape[0] == B, "page_table must be [B, max_pages]")
    _need(ctx_len.numel() == B and accept_len.numel() == B, "ctx_len / accept_len must be [B]")
    _need(emitted.numel() == B * (K + 1), "emitted must hold K+1 tokens per sequence")


def attn_dims(q: torch.Tensor, k_pages: torch.Tensor, page_table: torch.Tensor,
              softmax_scale: float = 0.0, flags: int = 0) -> AttnDims:
    """Geometry of one verify-attention call from q [B,R,Hq,D], the layer's
    pool [num_pages,Hkv,P,D] and the page table [B,max_pages]."""
    B, R, Hq, D = q.shape
    num_pages, Hkv, P, D2 = k_pages.shape[-4:]
    assert D2 == D
    return AttnDims(B, R, Hq, Hkv, D, P, page_table.shape[1], num_pages, softmax_scale, flags)


def num_sms() -> int:
    return load_library().cospec_num_sms()


ATTN_MMA_SYNC, ATTN_TCGEN05 = 0, 1
ATTN_KERNEL_NAMES = {ATTN_MMA_SYNC: "mma.sync", ATTN_TCGEN05: "tcgen05"}


def verify_attn_plan(q, k_pages, page_table, max_ctx: int, kv_stable: bool = False):
    """(kernel, splits) cospec_verify_attn would use for these tensors (and
    the stable-cache flag, which the plan of small batches depends on)."""
    dims = attn_dims(q, k_pages, page_table, flags=ATTN_KV_STABLE if kv_stable else 0)
    kernel, splits = ctypes.c_int(), ctypes.c_int()
    _check(load_library().cospec_verify_attn_plan(ctypes.byref(dims), int(max_ctx),
                                                  ctypes.byref(kernel), ctypes.byref(splits)))
    return kernel.value, splits.value


def verify_attn_plan_model(dims: AttnDims, max_ctx: int, num_sms: int, resident):
    """(kernel, splits) of cospec_verify_attn_plan_model: the plan for a
    device of ``num_sms`` SMs whose residency is ``resident(kernel, rows,
    block_rows, splits)`` -> clusters resident at once.  Host only."""
    cb = RESIDENT_FN(lambda k, r, kb, s, _user: int(resident(k, r, kb, s)))
    kernel, splits = ctypes.c_int(), ctypes.c_int()
    _check(load_library().cospec_verify_attn_plan_model(ctypes.byref(dims), int(max_ctx),
                                                        int(num_sms), cb, None,
                                                        ctypes.byref(kernel), ctypes.byref(splits)))
    return kernel.value, splits.value


def verify_attn(q, k_blk, v_blk, k_pages, v_pages, page_table, ctx_len, out, max_ctx,
                softmax_scale: float = 0.0, stream=None, kv_stable: bool = False,
                block_full: bool = False) -> torch.Tensor:
    """Verify attention of one layer (Sec. 3.1, Eq. 2).  See include/cospec.h.
    ``kv_stable``: the kernel queued just before writes neither ctx_len, the
    page table nor the cached pages (COSPEC_ATTN_KV_STABLE).  ``block_full``:
    block rows see the whole block (the arbitrator's draft/target region,
    Sec. 3.3; COSPEC_ATTN_BLOCK_FULL)."""
    for t, n in ((q, "q"), (k_blk, "k_blk"), (v_blk, "v_blk"), (k_pages, "k_pages"),
                 (v_pages, "v_pages"), (out, "out")):
        _req(t, torch.bfloat16, n)
    _req(page_table, torch.int32, "page_table", 2)
    _req(ctx_len, torch.int32, "ctx_len", 1)
    check_attn_shapes(q, k_blk, v_blk, k_pages, v_pages, page_table, ctx_len, out)
    _same_device(q, k_blk, v_blk, k_pages, v_pages, page_table, ctx_len, out)
    dims = attn_dims(q, k_pages, page_table, softmax_scale,
                     (ATTN_KV_STABLE if kv_stable else 0) | (ATTN_BLOCK_FULL if block_full else 0))
    _check(load_library().cospec_verify_attn(
        ctypes.byref(dims), int(max_ctx), _ptr(q), _ptr(k_blk), _ptr(v_blk), _ptr(k_pages),
        _ptr(v_pages), _ptr(page_table), _ptr(ctx_len), _ptr(out), _stream(stream)))
    return out


def lmhead_workspace_bytes(M: int, d: int, V: int) -> int:
    return load_library().cospec_lmhead_workspace(M, d, V)


def new_lmhead_workspace(M: int, d: int, V: int, device="cuda") -> torch.Tensor:
    return torch.empty(lmhead_workspace_bytes(M, d, V), dtype=torch.uint8, device=device)


def lmhead_argmax_features(hidden, w, draft_for_row, argmax, stats, ws, stream=None):
    """LM head + argmax + statistics (Eq. 2, Eq. 23).  stats [M,5] = (max,
    second, lse, entropy, draft logit)."""
    _req(hidden, torch.bfloat16, "hidden", 2)
    _req(w, torch.bfloat16, "w", 2)
    _req(draft_for_row, torch.int32, "draft_for_row", 1)
    _req(argmax, torch.int32, "argmax", 1)
    _req(stats, torch.float32, "stats", 2)
    _req(ws, torch.uint8, "ws", 1)
    M, d = hidden.shape
    V = w.shape[0]
    if w.shape[1] != d or draft_for_row.numel() != M or argmax.numel() != M or tuple(stats.shape) != (M, 5):
        raise ValueError("inconsistent LM-head shapes")
    _same_device(hidden, w, draft_for_row, argmax, stats, ws)
    _check(load_library().cospec_lmhead_argmax_features(
        M, d, V, _ptr(hidden), _ptr(w), _ptr(draft_for_row), _ptr(argmax), _ptr(stats), _ptr(ws),
        ws.numel(), _stream(stream)))
    return argmax, stats


def lmhead_sample_features(hidden, w, draft_for_row, temperature: float, seed, sample, stats, ws,
                           stream=None):
    """Stochastic-decoding LM head (Sec. 3.1, App. C.3): sample [M] is a
    Gumbel-max draw from softmax(x / T) with Philox4x32-10 noise keyed by the
    int64 device scalar ``seed`` (read when the kernel runs); stats as in
    lmhead_argmax_features."""
    _req(hidden, torch.bfloat16, "hidden", 2)
    _req(w, torch.bfloat16, "w", 2)
    _req(draft_for_row, torch.int32, "draft_for_row", 1)
    _req(sample, torch.int32, "sample", 1)
    _req(stats, torch.float32, "stats", 2)
    _req(ws, torch.uint8, "ws", 1)
    _req(seed, torch.int64, "seed")
    if seed.numel() != 1:
        raise ValueError("seed must hold one value")
    M, d = hidden.shape
    V = w.shape[0]
    if w.shape[1] != d or draft_for_row.numel() != M or sample.numel() != M or tuple(stats.shape) != (M, 5):
        raise ValueError("inconsistent LM-head shapes")
    _same_device(hidden, w, draft_for_row, seed, sample, stats, ws)
    _check(load_library().cospec_lmhead_sample_features(
        M, d, V, _ptr(hidden), _ptr(w), _ptr(draft_for_row), float(temperature), _ptr(seed),
        _ptr(sample), _ptr(stats), _ptr(ws), ws.numel(), _stream(stream)))
    return sample, stats


def lmhead_logits_features(hidden, w, draft_for_row, temperature: float, argmax, stats, logits,
                           ws, stream=None):
    """LM head for speculative sampling at temperature T: logits [M, V] fp32
    receives x / T, stats [M, 5] the statistics of x / T, argmax [M] the
    argmax."""
    _req(hidden, torch.bfloat16, "hidden", 2)
    _req(w, torch.bfloat16, "w", 2)
    _req(draft_for_row, torch.int32, "draft_for_row", 1)
    _req(argmax, torch.int32, "argmax", 1)
    _req(stats, torch.float32, "stats", 2)
    _req(logits, torch.float32, "logits", 2)
    _req(ws, torch.uint8, "ws", 1)
    M, d = hidden.shape
    V = w.shape[0]
    if (w.shape[1] != d or draft_for_row.numel() != M or argmax.numel() != M
            or tuple(stats.shape) != (M, 5) or tuple(logits.shape) != (M, V)):
        raise ValueError("inconsistent LM-head shapes")
    _same_device(hidden, w, draft_for_row, argmax, stats, logits, ws)
    _check(load_library().cospec_lmhead_logits_features(
        M, d, V, _ptr(hidden), _ptr(w), _ptr(draft_for_row), float(temperature), _ptr(argmax),
        _ptr(stats), _ptr(logits), _ptr(ws), ws.numel(), _stream(stream)))
    return argmax, stats, logits


def new_sps_workspace(B: int, device="cuda") -> torch.Tensor:
    return torch.empty(max(1, int(load_library().cospec_sps_workspace(B))), dtype=torch.uint8,
                       device=device)


def sps_accept(draft, stats, logits, q, seed, target, accept, ratio, ws, stream=None):
    """Speculative-sampling acceptance (the exact-match baseline at a
    temperature): draft [B, K], stats [B*(K+1), 5] and logits [B*(K+1), V]
    of x / T, q [B, K, V] the draft's distributions, seed an int64 device
    scalar; fills target [B, K+1], accept [B, K], ratio [B, K]."""
    _req(draft, torch.int32, "draft", 2)
    _req(stats, torch.float32, "stats", 2)
    _req(logits, torch.float32, "logits", 2)
    _req(q, torch.float32, "q", 3)
    _req(seed, torch.int64, "seed")
    _req(target, torch.int32, "target")
    _req(accept, torch.uint8, "accept")
    _req(ratio, torch.float32, "ratio")
    _req(ws, torch.uint8, "ws", 1)
    B, K = draft.shape
    R = K + 1
    V = logits.shape[1]
    if (seed.numel() != 1 or tuple(stats.shape) != (B * R, 5) or logits.shape[0] != B * R
            or tuple(q.shape) != (B, K, V) or target.numel() != B * R or accept.numel() != B * K
            or ratio.numel() != B * K):
        raise ValueError("inconsistent speculative-sampling shapes")
    _same_device(draft, stats, logits, q, seed, target, accept, ratio, ws)
    _check(load_library().cospec_sps_accept(
        B, K, V, _ptr(draft), _ptr(stats), _ptr(logits), _ptr(q), _ptr(seed), _ptr(target),
        _ptr(accept), _ptr(ratio), _ptr(ws), ws.numel(), _stream(stream)))
    return target, accept, ratio


def lmhead_argmax_features_noalloc(hidden, w, draft_for_row, argmax, stats, stream=None):
    """The LM-head call without a workspace, for callers that cannot allocate
    device memory: partials go to a fixed scratch array inside the library
    (at most 512 rows per call; calls must not overlap on the GPU)."""
    _req(hidden, torch.bfloat16, "hidden", 2)
    _req(w, torch.bfloat16, "w", 2)
    _req(draft_for_row, torch.int32, "draft_for_row", 1)
    _req(argmax, torch.int32, "argmax", 1)
    _req(stats, torch.float32, "stats", 2)
    M, d = hidden.shape
    V = w.shape[0]
    if w.shape[1] != d or draft_for_row.numel() != M or argmax.numel() != M or tuple(stats.shape) != (M, 5):
        raise ValueError("inconsistent LM-head shapes")
    _same_device(hidden, w, draft_for_row, argmax, stats)
    _check(load_library().cospec_lmhead_argmax_features_noalloc(
        M, d, V, _ptr(hidden), _ptr(w), _ptr(draft_for_row), _ptr(argmax), _ptr(stats),
        _stream(stream)))
    return argmax, stats


def rl_advantages(group_off, correct, round_off, match, accept, ell, params: RLParams = None,
                  ratio=None, p_new=None, p_ref=None, stream=None) -> dict:
    """RL-stage rewards and advantages (Sec. 3.4).  Inputs are CUDA tensors:
    group_off int32 [G+1], correct uint8 [M], round_off int32 [M+1],
    match / accept uint8 [R, K], ell float32 [R, K]; optional ratio / p_new /
    p_ref float32 [R, K] for the objective.  Returns the output tensors."""
    params = params if params is not None else RLParams()
    _req(group_off, torch.int32, "group_off", 1)
    _req(round_off, torch.int32, "round_off", 1)
    _req(correct, torch.uint8, "correct", 1)
    _req(match, torch.uint8, "match", 2)
    _req(accept, torch.uint8, "accept", 2)
    _req(ell, torch.float32, "ell", 2)
    G, M = group_off.numel() - 1, correct.numel()
    R, K = match.shape
    if round_off.numel() != M + 1 or tuple(accept.shape) != (R, K) or tuple(ell.shape) != (R, K):
        raise ValueError("inconsistent RL shapes")
    obj = [t for t in (ratio, p_new, p_ref) if t is not None]
    for t, n in zip(obj, ("ratio", "p_new", "p_ref")):
        _req(t, torch.float32, n, 2)
        if tuple(t.shape) != (R, K):
            raise ValueError(f"{n} must be [R, K]")
    _same_device(group_off, correct, round_off, match, accept, ell, *obj)
    dev = match.device
    out = dict(g=torch.empty((R, K), dtype=torch.float32, device=dev),
               eff=torch.empty((R, K), dtype=torch.uint8, device=dev),
               rho=torch.empty(R, dtype=torch.float32, device=dev),
               J=torch.empty(M, dtype=torch.float32, device=dev),
               Jbar=torch.empty(M, dtype=torch.float32, device=dev),
               adv=torch.empty(M, dtype=torch.float32, device=dev),
               adv_dec=torch.empty((R, K), dtype=torch.float32, device=dev))
    loss = torch.empty(4, dtype=torch.float32, device=dev) if obj else None
    lib = load_library()
    ws = torch.empty(lib.cospec_rl_workspace(G, M), dtype=torch.uint8, device=dev)
    _check(lib.cospec_rl_advantages(
        G, M, R, K, _ptr(group_off), _ptr(correct), _ptr(round_off), _ptr(match), _ptr(accept),
        _ptr(ell), ctypes.byref(params), _ptr(ratio), _ptr(p_new), _ptr(p_ref), _ptr(out["g"]),
        _ptr(out["eff"]), _ptr(out["rho"]), _ptr(out["J"]), _ptr(out["Jbar"]), _ptr(out["adv"]),
        _ptr(out["adv_dec"]), _ptr(loss), _ptr(ws), ws.numel(), _stream(stream)))
    if loss is not None:
        out["loss"] = loss
    return out


def arbitrate(draft, argmax, stats, w1, b1, w2, b2: float, lam: float, mode: int, p_out, accept,
              stream=None):
    """Mismatch arbitration (Eq. 3, Eq. 13-14, Eq. 17).  draft [B,K],
    argmax [B,K+1], stats [B,K+1,5]; p_out [B,K] float32, accept [B,K] uint8."""
    _req(draft, torch.int32, "draft", 2)
    _req(argmax, torch.int32, "argmax")
    _req(stats, torch.float32, "stats")
    _req(p_out, torch.float32, "p_out")
    _req(accept, torch.uint8, "accept")
    B, K = draft.shape
    H = 0
    if mode == POLICY_MLP:
        for t, n in ((w1, "w1"), (b1, "b1"), (w2, "w2")):
            _req(t, torch.float32, n)
        H = w1.shape[0]
    check_arbitrate_shapes(draft, argmax, stats, w1, b1, w2, mode, p_out, accept)
    _same_device(draft, argmax, stats, p_out, accept,
                 *((w1, b1, w2) if mode == POLICY_MLP else ()))
    _check(load_library().cospec_arbitrate(
        B, K, _ptr(draft), _ptr(argmax), _ptr(stats), H, _ptr(w1) if mode == 0 else None,
        _ptr(b1) if mode == 0 else None, _ptr(w2) if mode == 0 else None, float(b2), float(lam),
        int(mode), _ptr(p_out), _ptr(accept), _stream(stream)))
    return p_out, accept


def accept_commit(draft, argmax, accept, k_blk, v_blk, k_pages, v_pages, page_table, ctx_len,
                  accept_len, emitted, stream=None):
    """Accepted length / emitted tokens (Eq. 15) and KV commit.
    k_blk, v_blk [L,B,R,Hkv,D]; pools [L,num_pages,Hkv,P,D] (any layer stride)."""
    _req(draft, torch.int32, "draft", 2)
    _req(argmax, torch.int32, "argmax")
    _req(accept, torch.uint8, "accept")
    for t, n in ((k_blk, "k_blk"), (v_blk, "v_blk")):
        _req(t, torch.bfloat16, n, 5)
    for t, n in ((k_pages, "k_pages"), (v_pages, "v_pages")):
        if t.dtype != torch.bfloat16 or not t.is_cuda or t.dim() != 5 or not t[0].is_contiguous():
            raise ValueError(f"{n}: expected bf16 CUDA [L,num_pages,Hkv,P,D] with contiguous layers")
    _req(page_table, torch.int32, "page_table", 2)
    _req(ctx_len, torch.int32, "ctx_len", 1)
    _req(accept_len, torch.int32, "accept_len", 1)
    _req(emitted, torch.int32, "emitted")
    check_commit_shapes(draft, argmax, accept, k_blk, v_blk, k_pages, v_pages, page_table,
                        ctx_len, accept_len, emitted)
    _same_device(draft, argmax, accept, k_blk, v_blk, k_pages, v_pages, page_table, ctx_len,
                 accept_len, emitted)
    B, K = draft.shape
    L = k_blk.shape[0]
    if k_pages.stride(0) != v_pages.stride(0):
        raise ValueError("k_pages / v_pages must hold their layers with the same stride")
    # A single pool standing for every layer receives layer 0's rows only (the
    # library rejects several layers committed into one pool: their writes
    # would race for the same cells).
    if k_pages.shape[0] == 1 and L > 1:
        L = 1
        k_blk, v_blk = k_blk[:1], v_blk[:1]
    layer_stride = int(k_pages.stride(0))
    dims = AttnDims(B, K + 1, 0, k_pages.shape[2], k_pages.shape[4], k_pages.shape[3],
                    page_table.shape[1], k_pages.shape[1], 0.0, 0)
    dims.num_q_heads = dims.num_kv_heads
    _check(load_library().cospec_accept_commit(
        B, K, L, ctypes.byref(dims), _ptr(draft), _ptr(argmax), _ptr(accept), _ptr(k_blk),
        _ptr(v_blk), _ptr(k_pages), _ptr(v_pages), layer_stride, _ptr(page_table),
        _ptr(ctx_len), _ptr(accept_len), _ptr(emitted), _stream(stream)))
    return accept_len, emitted


def get_device_error(stream=None) -> int:
    """Read and clear the device error word (synchronises the stream)."""
    flags = ctypes.c_int(0)
    st = load_library().cospec_get_device_error(ctypes.byref(flags), _stream(stream))
    if st not in (0, -5):
        _check(st)
    return flags.value
