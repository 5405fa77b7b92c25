"""ctypes binding of libgrpo.so (include/grpo.h), same names as the C ABI.

Argument marshalling only: every step of the computation runs in the
library's CUDA kernels.  PyTorch provides device memory and the current
stream.  Inputs may be CUDA tensors, or CPU tensors (preferably pinned): CPU
inputs are copied to the current CUDA device, the call runs there, and the
results are copied back to CPU tensors.

There is no fallback: if libgrpo.so is missing or the device is not a GB300
class GPU, the calls raise.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Tuple

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libgrpo.so")

GRPO_OK = 0
GRPO_ERR_INVALID_ARG = 1
GRPO_ERR_WORKSPACE = 2
GRPO_ERR_CUDA = 3
GRPO_ERR_DEVICE_CHECK = 4
GRPO_ERR_TIMEOUT = 5
GRPO_ERR_UNSUPPORTED = 6
GRPO_ERR_CAPACITY = 7
GRPO_WS_LOGPROBS = 0
GRPO_WS_LOSS = 1
GRPO_WS_LOGPROBS_HEADS = 2
GRPO_WS_SAMPLE = 3
GRPO_WS_LOSS_LOGITS = 4
GRPO_WS_SAMPLE_TOP_P = 5
GRPO_MAX_HEADS = 4

# name -> (restype, argtypes); mirrors include/grpo.h
_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_I32 = ctypes.c_int32
_F = ctypes.c_float
SIGNATURES = {
    "grpo_group_advantages": (ctypes.c_int, [_P, _I64, _I32, _F, _P, _P]),
    "grpo_token_logprobs": (ctypes.c_int, [_P, _P, _P, _P, _I64, _I32, _I64, _P, _P, ctypes.c_size_t, _P]),
    "grpo_loss_fwd_bwd": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _I64, _I64, _I32, _I64, _F, _F, _I32,
                                         _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "grpo_token_logprobs_heads": (ctypes.c_int, [_P, _P, _I32, _P, _P, _I64, _I32, _I64, _P, _P, ctypes.c_size_t,
                                                 _P]),
    "grpo_loss_fwd_bwd_norm": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _I64, _I64, _I32, _I64, _F, _F, _I32, _F,
                                              _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "grpo_loss_fwd_bwd_kl_clamp": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _I64, _I64, _I32, _I64, _F, _F, _I32,
                                                  _F, _F, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "grpo_loss_fwd_bwd_events": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _I64, _I64, _I32, _I64, _F, _F, _I32,
                                                _F, _P, _P, _P, _P, _I32, _P, ctypes.c_size_t, _P]),
    "grpo_vocab_chunk_cols": (ctypes.c_int64, [_I64]),
    "grpo_loss_fwd_bwd_to_host": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _I64, _I64, _I32, _I64, _F, _F, _I32,
                                                 _F, _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "grpo_loss_fwd_bwd_adamw": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _I64, _I64, _I32, _I64, _F, _F, _I32, _F,
                                               _F, _F, _F, _F, _F, _I64, _P, _P, _P, _P, _P, _P, _P,
                                               ctypes.c_size_t, _P]),
    "grpo_sample_tokens": (ctypes.c_int, [_P, _P, _P, _I64, _I32, _I64, _F, ctypes.c_uint64, ctypes.c_uint64, _P, _P,
                                          _P, ctypes.c_size_t, _P]),
    "grpo_sample_tokens_top_p": (ctypes.c_int, [_P, _P, _P, _I64, _I32, _I64, _F, _F, ctypes.c_uint64,
                                                ctypes.c_uint64, _P, _P, _P, ctypes.c_size_t, _P]),
    "grpo_gumbel_noise": (ctypes.c_int, [ctypes.c_uint64, ctypes.c_uint64, _I64, _I64, _I64, _P, _P]),
    "grpo_adamw_step": (ctypes.c_int, [_P, _P, _P, _P, _P, _I64, _F, _F, _F, _F, _F, _I64, _P]),
    "grpo_token_logprobs_noalloc": (ctypes.c_int, [_P, _P, _P, _P, _I64, _I32, _I64, _P, _P]),
    "grpo_noalloc_check_status": (ctypes.c_int, [_P]),
    "grpo_workspace_bytes": (ctypes.c_size_t, [_I64, _I32, _I64, _I32]),
    "grpo_workspace_bytes_rows": (ctypes.c_size_t, [_I64, _I64, _I32, _I64, _I32]),
    "grpo_loss_plan": (ctypes.c_int32, [_I64, _I32, _I64, ctypes.c_size_t, _P]),
    "grpo_check_device_status": (ctypes.c_int, [_P, _P]),
    "grpo_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "grpo_trace_enable": (ctypes.c_int, [_I32]),
    "grpo_trace_read": (ctypes.c_int32, [_P, _P, _P, _I32]),
}

_lib: Optional[ctypes.CDLL] = None


class GrpoError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


def open_library(path: str) -> ctypes.CDLL:
    """dlopen the library at `path` and declare its signatures; raises ImportError if absent."""
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with `python -m paper_2507_05687_gb300.build`")
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


def load() -> ctypes.CDLL:
    """The in-tree libgrpo.so (built by build.py), opened once per process."""
    global _lib
    if _lib is None:
        _lib = open_library(LIB_PATH)
    return _lib


def status_string(status: int) -> str:
    return load().grpo_status_string(int(status)).decode()


def _check(st: int, where: str) -> None:
    if st != GRPO_OK:
        raise GrpoError(st, where)


def _stream(device: torch.device) -> int:
    return torch.cuda.current_stream(device).cuda_stream


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _on_device(t: torch.Tensor, dev: torch.device, dtype: torch.dtype, name: str) -> torch.Tensor:
    if t.dtype != dtype:
        raise TypeError(f"{name}: expected {dtype}, got {t.dtype}")
    if t.device != dev:
        t = t.to(dev, non_blocking=True)
    return t.contiguous()


def _hidden(H: torch.Tensor, dev: torch.device) -> torch.Tensor:
    """H for the C call: left in page-locked host memory when it is there (the
    library's row gather then reads only the unmasked rows over the host link),
    else on `dev` (copied when it is elsewhere)."""
    if H.dtype != torch.bfloat16:
        raise TypeError(f"H: expected {torch.bfloat16}, got {H.dtype}")
    if not H.is_cuda and H.is_contiguous() and H.is_pinned():
        return H
    return _on_device(H, dev, torch.bfloat16, "H")


# Host tensors the device reads during a call (a page-locked H): each stays
# referenced until an event recorded after the call's work has completed, so
# that it cannot be freed or reused while the row gather still reads it.
_in_flight = []


def _keep_until_done(t: torch.Tensor, dev: torch.device) -> None:
    if t.is_cuda:
        return
    if not torch.cuda.is_current_stream_capturing():  # no event queries inside a graph capture
        while _in_flight and _in_flight[0][0].query():
            _in_flight.pop(0)
    ev = torch.cuda.Event()
    ev.record(torch.cuda.current_stream(dev))
    _in_flight.append((ev, t))


def _shape(t: torch.Tensor, shape, name: str) -> None:
    """The C ABI sees only pointers and sizes: a tensor of the wrong shape would
    be read or written past its end, so every shape is checked here."""
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: expected shape {tuple(shape)}, got {tuple(t.shape)}")


def _output(t: torch.Tensor, shape, dtype: torch.dtype, dev: torch.device, name: str) -> torch.Tensor:
    """A caller-given output is written in place: it must already be a dense
    tensor of the right shape, type and device (a copy would be written instead)."""
    if t.dtype != dtype or t.device != dev or not t.is_contiguous():
        raise ValueError(f"{name}: contiguous {dtype} on {dev} expected")
    _shape(t, shape, name)
    return t


def _workspace(ws: torch.Tensor, dev: torch.device) -> torch.Tensor:
    if ws.dtype != torch.uint8 or ws.device != dev or not ws.is_contiguous():
        raise ValueError(f"ws: contiguous uint8 on {dev} expected (see workspace())")
    return ws


def _target_device(*ts: torch.Tensor) -> Tuple[torch.device, bool]:
    for t in ts:
        if t.is_cuda:
            return t.device, False
    return torch.device("cuda", torch.cuda.current_device()), True


def _to_host(*ts: torch.Tensor, dst=None):
    """Host copies of device results (into `dst` host tensors when given,
    else new pinned ones); returns once they have landed."""
    outs = []
    for i, t in enumerate(ts):
        o = dst[i] if dst is not None else torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        o.copy_(t, non_blocking=True)
        outs.append(o)
    torch.cuda.current_stream(ts[0].device).synchronize()
    return outs[0] if len(outs) == 1 else tuple(outs)


def workspace_bytes(T: int, Hd: int, V: int, which: int) -> int:
    """grpo_workspace_bytes: scratch bytes the call `which` needs."""
    return int(load().grpo_workspace_bytes(int(T), int(Hd), int(V), int(which)))


def workspace_bytes_rows(T: int, max_valid: int, Hd: int, V: int, which: int) -> int:
    """grpo_workspace_bytes_rows: scratch bytes for batches with at most max_valid unmasked rows."""
    return int(load().grpo_workspace_bytes_rows(int(T), int(max_valid), int(Hd), int(V), int(which)))


def loss_plan(T: int, Hd: int, V: int, ws_bytes: int) -> Tuple[int, int]:
    """grpo_loss_plan: (1 if the loss calls keep the logits for the backward
    with a workspace of ws_bytes, else 0; the row capacity)."""
    rows = ctypes.c_int64(0)
    kept = int(load().grpo_loss_plan(int(T), int(Hd), int(V), int(ws_bytes), ctypes.byref(rows)))
    if kept < 0:
        raise GrpoError(GRPO_ERR_WORKSPACE, "grpo_loss_plan")
    return kept, int(rows.value)


def loss_workspace(T: int, Hd: int, V: int, device=None, max_valid: Optional[int] = None,
                   keep_logits: bool = False) -> torch.Tensor:
    """A workspace for the loss calls.  By default the plain one
    (GRPO_WS_LOSS): the backward recomputes the logits chunk by chunk and no
    [tokens x vocabulary] buffer exists.  keep_logits=True sizes it exactly
    for GRPO_WS_LOSS_LOGITS instead: the forward stores the fp32 logits and the
    backward reads them back (same results, bit for bit)."""
    which = GRPO_WS_LOSS_LOGITS if keep_logits else GRPO_WS_LOSS
    return workspace(T, Hd, V, which, device or "cuda", max_valid=max_valid)


def workspace(T: int, Hd: int, V: int, which: int, device=None, max_valid: Optional[int] = None) -> torch.Tensor:
    """A device byte tensor large enough for the call `which` (for batches with at
    most max_valid unmasked rows when given)."""
    n = workspace_bytes(T, Hd, V, which) if max_valid is None else workspace_bytes_rows(T, max_valid, Hd, V, which)
    if n == 0:
        raise GrpoError(GRPO_ERR_INVALID_ARG, "grpo_workspace_bytes")
    return torch.empty(n, dtype=torch.uint8, device=device or "cuda")


def group_advantages(rewards: torch.Tensor, G: int, eps: float = 1e-6,
                     out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """grpo_group_advantages: Eq. 2 per group of G consecutive responses."""
    dev, host = _target_device(rewards)
    r = _on_device(rewards, dev, torch.float32, "rewards").reshape(-1)
    adv = _output(out, r.shape, torch.float32, dev, "out") if out is not None else torch.empty_like(r)
    _check(load().grpo_group_advantages(_ptr(r), r.numel(), int(G), float(eps), _ptr(adv), _stream(dev)),
           "grpo_group_advantages")
    return _to_host(adv) if host else adv


def token_logprobs(H: torch.Tensor, W: torch.Tensor, targets: torch.Tensor, mask: torch.Tensor,
                   ws: Optional[torch.Tensor] = None, out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """grpo_token_logprobs: log softmax(H W^T) at the sampled tokens; padding rows give 0."""
    dev, host = _target_device(H, W)
    H = _hidden(H, dev)
    W = _on_device(W, dev, torch.bfloat16, "W")
    targets = _on_device(targets, dev, torch.int32, "targets")
    mask = _on_device(mask.view(torch.uint8) if mask.dtype == torch.bool else mask, dev, torch.uint8, "mask")
    T, Hd = H.shape
    V = W.shape[0]
    _shape(W, (V, Hd), "W")
    _shape(targets, (T,), "targets")
    _shape(mask, (T,), "mask")
    ws = workspace(T, Hd, V, GRPO_WS_LOGPROBS, dev) if ws is None else _workspace(ws, dev)
    logp = _output(out, (T,), torch.float32, dev, "out") if out is not None else \
        torch.empty(T, dtype=torch.float32, device=dev)
    _check(load().grpo_token_logprobs(_ptr(H), _ptr(W), _ptr(targets), _ptr(mask), T, Hd, V, _ptr(logp),
                                      _ptr(ws), ws.numel(), _stream(dev)), "grpo_token_logprobs")
    _keep_until_done(H, dev)
    return _to_host(logp) if host else logp


def token_logprobs_heads(H: torch.Tensor, W_heads, targets: torch.Tensor, mask: torch.Tensor,
                         ws: Optional[torch.Tensor] = None, out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """grpo_token_logprobs_heads: log-probs under each head in W_heads (policy,
    old, reference ...); returns [n_heads, T] fp32, 0 on padding rows."""
    W_heads = list(W_heads)
    dev, host = _target_device(H, *W_heads)
    H = _hidden(H, dev)
    W_heads = [_on_device(w, dev, torch.bfloat16, f"W_heads[{i}]") for i, w in enumerate(W_heads)]
    targets = _on_device(targets, dev, torch.int32, "targets")
    mask = _on_device(mask.view(torch.uint8) if mask.dtype == torch.bool else mask, dev, torch.uint8, "mask")
    T, Hd = H.shape
    V = W_heads[0].shape[0]
    for i, w in enumerate(W_heads):
        _shape(w, (V, Hd), f"W_heads[{i}]")
    _shape(targets, (T,), "targets")
    _shape(mask, (T,), "mask")
    ws = workspace(T, Hd, V, GRPO_WS_LOGPROBS_HEADS, dev) if ws is None else _workspace(ws, dev)
    logp = _output(out, (len(W_heads), T), torch.float32, dev, "out") if out is not None else \
        torch.empty(len(W_heads), T, dtype=torch.float32, device=dev)
    ptrs = (ctypes.c_void_p * len(W_heads))(*[w.data_ptr() for w in W_heads])
    _check(load().grpo_token_logprobs_heads(_ptr(H), ptrs, len(W_heads), _ptr(targets), _ptr(mask), T, Hd, V,
                                            _ptr(logp), _ptr(ws), ws.numel(), _stream(dev)),
           "grpo_token_logprobs_heads")
    _keep_until_done(H, dev)
    return _to_host(logp) if host else logp


def sample_tokens(H: torch.Tensor, W: torch.Tensor, mask: torch.Tensor, temperature: float = 1.0, seed: int = 0,
                  offset: int = 0, ws: Optional[torch.Tensor] = None, out=None):
    """grpo_sample_tokens: Gumbel-max draw from softmax(H W^T / temperature) at
    the unmasked rows; returns (tokens int32 [T] (-1 masked), logp fp32 [T])."""
    dev, host = _target_device(H, W)
    H = _hidden(H, dev)
    W = _on_device(W, dev, torch.bfloat16, "W")
    mask = _on_device(mask.view(torch.uint8) if mask.dtype == torch.bool else mask, dev, torch.uint8, "mask")
    T, Hd = H.shape
    V = W.shape[0]
    _shape(W, (V, Hd), "W")
    _shape(mask, (T,), "mask")
    ws = workspace(T, Hd, V, GRPO_WS_SAMPLE, dev) if ws is None else _workspace(ws, dev)
    if out is None:
        out = (torch.empty(T, dtype=torch.int32, device=dev), torch.empty(T, dtype=torch.float32, device=dev))
    tok = _output(out[0], (T,), torch.int32, dev, "out[0]")
    logp = _output(out[1], (T,), torch.float32, dev, "out[1]")
    _check(load().grpo_sample_tokens(_ptr(H), _ptr(W), _ptr(mask), T, Hd, V, float(temperature),
                                     int(seed) & (2 ** 64 - 1), int(offset) & (2 ** 64 - 1), _ptr(tok), _ptr(logp),
                                     _ptr(ws), ws.numel(), _stream(dev)), "grpo_sample_tokens")
    _keep_until_done(H, dev)
    return _to_host(tok, logp) if host else (tok, logp)


def sample_tokens_top_p(H: torch.Tensor, W: torch.Tensor, mask: torch.Tensor, temperature: float = 1.0,
                        top_p: float = 1.0, seed: int = 0, offset: int = 0, ws: Optional[torch.Tensor] = None,
                        out=None):
    """grpo_sample_tokens_top_p: the draw of sample_tokens restricted to the
    nucleus of softmax(H W^T / temperature) (the most probable tokens whose mass
    reaches top_p); returns (tokens int32 [T] (-1 masked), logp fp32 [T] under
    the untruncated distribution)."""
    dev, host = _target_device(H, W)
    H = _hidden(H, dev)
    W = _on_device(W, dev, torch.bfloat16, "W")
    mask = _on_device(mask.view(torch.uint8) if mask.dtype == torch.bool else mask, dev, torch.uint8, "mask")
    T, Hd = H.shape
    V = W.shape[0]
    _shape(W, (V, Hd), "W")
    _shape(mask, (T,), "mask")
    ws = workspace(T, Hd, V, GRPO_WS_SAMPLE_TOP_P, dev) if ws is None else _workspace(ws, dev)
    if out is None:
        out = (torch.empty(T, dtype=torch.int32, device=dev), torch.empty(T, dtype=torch.float32, device=dev))
    tok = _output(out[0], (T,), torch.int32, dev, "out[0]")
    logp = _output(out[1], (T,), torch.float32, dev, "out[1]")
    _check(load().grpo_sample_tokens_top_p(_ptr(H), _ptr(W), _ptr(mask), T, Hd, V, float(temperature),
                                           float(top_p), int(seed) & (2 ** 64 - 1), int(offset) & (2 ** 64 - 1),
                                           _ptr(tok), _ptr(logp), _ptr(ws), ws.numel(), _stream(dev)),
           "grpo_sample_tokens_top_p")
    _keep_until_done(H, dev)
    return _to_host(tok, logp) if host else (tok, logp)


def loss_fwd_bwd(H: torch.Tensor, W: torch.Tensor, targets: torch.Tensor, mask: torch.Tensor,
                 old_logp: torch.Tensor, ref_logp: torch.Tensor, adv: torch.Tensor,
                 n_resp: int, L: int, clip_eps: float = 0.2, beta: float = 0.04, agg_mode: int = 0,
                 ws: Optional[torch.Tensor] = None,
                 out: Optional[Tuple[torch.Tensor, torch.Tensor, torch.Tensor]] = None, norm: float = 0.0,
                 kl_clamp: Optional[float] = None, chunk_events: Optional[list] = None):
    """grpo_loss_fwd_bwd (norm == 0) / grpo_loss_fwd_bwd_norm (norm > 0, a global
    N_valid or n_resp) / grpo_loss_fwd_bwd_kl_clamp (kl_clamp given, a cap on the
    per-token KL value) / grpo_loss_fwd_bwd_events (chunk_events: torch.cuda.Event
    per vocabulary chunk, recorded when that chunk's dW rows are written):
    returns (loss [1] fp32, dH [T, Hd] fp32, dW [V, Hd] fp32).
    `out` may be device tensors (written in place) or host tensors, preferably
    pinned (the results are copied there before the call returns)."""
    dev, host = _target_device(H, W)
    H = _hidden(H, dev)
    W = _on_device(W, dev, torch.bfloat16, "W")
    targets = _on_device(targets, dev, torch.int32, "targets")
    mask = _on_device(mask.view(torch.uint8) if mask.dtype == torch.bool else mask, dev, torch.uint8, "mask")
    old_logp = _on_device(old_logp, dev, torch.float32, "old_logp")
    ref_logp = _on_device(ref_logp, dev, torch.float32, "ref_logp")
    adv = _on_device(adv, dev, torch.float32, "adv")
    T, Hd = H.shape
    V = W.shape[0]
    if T != int(n_resp) * int(L):
        raise ValueError(f"H has {T} rows, n_resp * L = {int(n_resp) * int(L)}")
    _shape(W, (V, Hd), "W")
    for name, t in (("targets", targets), ("mask", mask), ("old_logp", old_logp), ("ref_logp", ref_logp)):
        _shape(t, (T,), name)
    _shape(adv, (int(n_resp),), "adv")
    ws = loss_workspace(T, Hd, V, dev) if ws is None else _workspace(ws, dev)
    host_out = None
    if out is not None and not out[0].is_cuda:
        host_out, out = out, None  # results land in the caller's host buffers
        for name, t, shp in (("out[0]", host_out[0], (1,)), ("out[1]", host_out[1], (T, Hd)),
                             ("out[2]", host_out[2], (V, Hd))):
            if t.dtype != torch.float32 or t.is_cuda or not t.is_contiguous():
                raise ValueError(f"{name}: contiguous fp32 host tensor expected")
            _shape(t, shp, name)
    if out is None:
        out = (torch.empty(1, dtype=torch.float32, device=dev),
               torch.empty(T, Hd, dtype=torch.float32, device=dev),
               torch.empty(V, Hd, dtype=torch.float32, device=dev))
    loss = _output(out[0], (1,), torch.float32, dev, "out[0]")
    dH = _output(out[1], (T, Hd), torch.float32, dev, "out[1]")
    dW = _output(out[2], (V, Hd), torch.float32, dev, "out[2]")
    lib = load()
    common = (_ptr(H), _ptr(W), _ptr(targets), _ptr(mask), _ptr(old_logp), _ptr(ref_logp), _ptr(adv), int(n_resp),
              int(L), Hd, V, float(clip_eps), float(beta), int(agg_mode))
    tail = (_ptr(loss), _ptr(dH), _ptr(dW), _ptr(ws), ws.numel(), _stream(dev))
    if host_out is not None and host_out[2].is_pinned() and kl_clamp is None and chunk_events is None:
        # dW streams to the caller's pinned buffer chunk by chunk while the backward runs
        _check(lib.grpo_loss_fwd_bwd_to_host(*common, float(norm), _ptr(loss), _ptr(dH), _ptr(dW),
                                             _ptr(host_out[2]), _ptr(ws), ws.numel(), _stream(dev)),
               "grpo_loss_fwd_bwd_to_host")
        _keep_until_done(H, dev)
        lh, dHh = _to_host(loss, dH, dst=host_out[:2])
        return lh, dHh, host_out[2]
    if chunk_events is not None:
        if kl_clamp is not None:
            raise ValueError("chunk_events and kl_clamp are separate entry points")
        stream = torch.cuda.current_stream(dev)
        for ev in chunk_events:
            if not ev.cuda_event:
                ev.record(stream)  # torch creates the CUDA event on its first record
        evs = (ctypes.c_void_p * max(1, len(chunk_events)))(*[ev.cuda_event for ev in chunk_events])
        _check(lib.grpo_loss_fwd_bwd_events(*common, float(norm), _ptr(loss), _ptr(dH), _ptr(dW), evs,
                                            len(chunk_events), _ptr(ws), ws.numel(), _stream(dev)),
               "grpo_loss_fwd_bwd_events")
    elif kl_clamp is not None:
        _check(lib.grpo_loss_fwd_bwd_kl_clamp(*common, float(norm), float(kl_clamp), *tail),
               "grpo_loss_fwd_bwd_kl_clamp")
    elif norm:
        _check(lib.grpo_loss_fwd_bwd_norm(*common, float(norm), *tail), "grpo_loss_fwd_bwd_norm")
    else:
        _check(lib.grpo_loss_fwd_bwd(*common, *tail), "grpo_loss_fwd_bwd")
    _keep_until_done(H, dev)
    if host or host_out is not None:
        return _to_host(loss, dH, dW, dst=host_out)
    return loss, dH, dW


def loss_fwd_bwd_adamw(H: torch.Tensor, W: torch.Tensor, targets: torch.Tensor, mask: torch.Tensor,
                       old_logp: torch.Tensor, ref_logp: torch.Tensor, adv: torch.Tensor, n_resp: int, L: int,
                       W_master: torch.Tensor, exp_avg: torch.Tensor, exp_avg_sq: torch.Tensor, step: int,
                       lr: float = 1e-6, betas=(0.9, 0.999), eps: float = 1e-8, weight_decay: float = 0.01,
                       clip_eps: float = 0.2, beta: float = 0.04, agg_mode: int = 0, norm: float = 0.0,
                       W_out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                       out: Optional[Tuple[torch.Tensor, torch.Tensor]] = None):
    """grpo_loss_fwd_bwd_adamw: loss and dH as loss_fwd_bwd; the LM-head gradient
    is consumed by an AdamW step on W_master / exp_avg / exp_avg_sq (device fp32,
    in place) and W_out (bf16, default W itself).  Returns (loss, dH)."""
    dev = W.device
    if not (H.is_cuda and W.is_cuda and W_master.is_cuda and exp_avg.is_cuda and exp_avg_sq.is_cuda):
        raise ValueError("loss_fwd_bwd_adamw takes device tensors")
    H = _on_device(H, dev, torch.bfloat16, "H")
    targets = _on_device(targets, dev, torch.int32, "targets")
    mask = _on_device(mask.view(torch.uint8) if mask.dtype == torch.bool else mask, dev, torch.uint8, "mask")
    old_logp = _on_device(old_logp, dev, torch.float32, "old_logp")
    ref_logp = _on_device(ref_logp, dev, torch.float32, "ref_logp")
    adv = _on_device(adv, dev, torch.float32, "adv")
    for name, t in (("W_master", W_master), ("exp_avg", exp_avg), ("exp_avg_sq", exp_avg_sq)):
        if t.dtype != torch.float32 or not t.is_contiguous() or t.shape != W.shape:
            raise ValueError(f"{name}: contiguous fp32 [V, Hd] expected")
    W_out = W if W_out is None else W_out
    T, Hd = H.shape
    V = W.shape[0]
    if T != int(n_resp) * int(L):
        raise ValueError(f"H has {T} rows, n_resp * L = {int(n_resp) * int(L)}")
    if W.dtype != torch.bfloat16 or not W.is_contiguous():
        raise ValueError("W: contiguous bf16 expected")
    _shape(W, (V, Hd), "W")
    _output(W_out, (V, Hd), torch.bfloat16, dev, "W_out")
    for name, t in (("targets", targets), ("mask", mask), ("old_logp", old_logp), ("ref_logp", ref_logp)):
        _shape(t, (T,), name)
    _shape(adv, (int(n_resp),), "adv")
    ws = loss_workspace(T, Hd, V, dev) if ws is None else _workspace(ws, dev)
    if out is None:
        out = (torch.empty(1, dtype=torch.float32, device=dev), torch.empty(T, Hd, dtype=torch.float32, device=dev))
    loss = _output(out[0], (1,), torch.float32, dev, "out[0]")
    dH = _output(out[1], (T, Hd), torch.float32, dev, "out[1]")
    _check(load().grpo_loss_fwd_bwd_adamw(
        _ptr(H), _ptr(W), _ptr(targets), _ptr(mask), _ptr(old_logp), _ptr(ref_logp), _ptr(adv), int(n_resp), int(L),
        Hd, V, float(clip_eps), float(beta), int(agg_mode), float(norm), float(lr), float(betas[0]), float(betas[1]),
        float(eps), float(weight_decay), int(step), _ptr(W_master), _ptr(exp_avg), _ptr(exp_avg_sq), _ptr(W_out),
        _ptr(loss), _ptr(dH), _ptr(ws), ws.numel(), _stream(dev)), "grpo_loss_fwd_bwd_adamw")
    return loss, dH


def adamw_step(W_master: torch.Tensor, exp_avg: torch.Tensor, exp_avg_sq: torch.Tensor, grad: torch.Tensor,
               W_out: torch.Tensor, step: int, lr: float = 1e-6, betas=(0.9, 0.999), eps: float = 1e-8,
               weight_decay: float = 0.01) -> None:
    """grpo_adamw_step: one AdamW step in place over contiguous fp32 device tensors."""
    n = W_master.numel()
    dev = W_master.device
    for name, t in (("W_master", W_master), ("exp_avg", exp_avg), ("exp_avg_sq", exp_avg_sq), ("grad", grad)):
        if t.numel() != n or t.dtype != torch.float32 or not t.is_contiguous() or t.device != dev or not t.is_cuda:
            raise ValueError(f"{name}: contiguous fp32 device tensor with W_master's size expected")
    if W_out.numel() != n or W_out.dtype != torch.bfloat16 or not W_out.is_contiguous() or W_out.device != dev:
        raise ValueError("W_out: contiguous bf16 with W_master's size expected")
    _check(load().grpo_adamw_step(_ptr(W_master), _ptr(exp_avg), _ptr(exp_avg_sq), _ptr(grad), _ptr(W_out), n,
                                  float(lr), float(betas[0]), float(betas[1]), float(eps), float(weight_decay),
                                  int(step), _stream(W_master.device)), "grpo_adamw_step")


def vocab_chunk_cols(V: int) -> int:
    """grpo_vocab_chunk_cols: dW rows per backward chunk (chunk c = rows c*cols ..)."""
    return int(load().grpo_vocab_chunk_cols(int(V)))


def gumbel_noise(row0: int, rows: int, cols: int, seed: int, offset: int = 0, device=None) -> torch.Tensor:
    """grpo_gumbel_noise: the fp32 noise grpo_sample_tokens adds to z / temperature at
    token positions row0 .. row0 + rows - 1 and vocabulary ids 0 .. cols - 1."""
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    out = torch.empty(rows, cols, dtype=torch.float32, device=dev)
    _check(load().grpo_gumbel_noise(int(seed) & (2**64 - 1), int(offset) & (2**64 - 1), int(row0), int(rows),
                                    int(cols), _ptr(out), _stream(dev)), "grpo_gumbel_noise")
    return out


def check_device_status(ws: torch.Tensor) -> int:
    """grpo_check_device_status: syncs the current stream and returns the status code."""
    return int(load().grpo_check_device_status(_ptr(ws), _stream(ws.device)))
