"""GB300-native BD-LRU scan (RecBLR, arXiv 2406.12580, Sec. 3.2-3.3).

Python front end of the C-ABI library ``libblr.so`` (declared in
``include/blr.h``). The functions named like the C entry points only marshal
arguments: they take CUDA tensors (or raw device pointers as ints), check
that tensors live on the current CUDA device, and call the library on the
current torch stream. Every step of the scan runs in the library's kernels;
there is no CPU path.

    desc = Desc(B, L, D, io=BLR_F32, c=1.0)
    ws = torch.empty(blr_workspace_bytes(desc), dtype=torch.uint8, device="cuda")
    blr_scan_fwd(desc, x, gate_logits, lam, h0, h, h_last, ws)
    blr_scan_bwd(desc, dh, dh_last, x, gate_logits, lam, h0, dx, dgate_logits, dlam, dh0, ws)
    blr_step(B, D, BLR_F32, 1.0, h_prev, x_t, gate_logits_t, lam, h_t)
    blr_steps(B, K, D, BLR_BF16, BLR_BF16, 1.0, h_prev, x, gate_logits, lam, h_out, h_seq)

The gated recurrent layer's merge y = h SiLU(z) (Alg. 1) fused into the scan:

    blr_scan_fwd_gated(desc, x, gate_logits, lam, h0, z, y, h_last, ws)
    blr_scan_bwd_gated(desc, dy, dh_last, x, gate_logits, lam, h0, z, dx, dgate_logits, dz,
                       dlam, dh0, ws)

``BDLRUScan`` wraps the forward and backward in a torch.autograd.Function.
"""
from __future__ import annotations

import ctypes

from ._lib import (BLR_BF16, BLR_ERR_CUDA, BLR_ERR_INVALID_ARG, BLR_ERR_TIMEOUT,  # noqa: F401
                   BLR_ERR_UNSUPPORTED, BLR_ERR_WORKSPACE, BLR_F32, BLR_OK, blr_desc, load)

__all__ = [
    "BLR_F32", "BLR_BF16", "Desc", "BLRError", "blr_workspace_bytes", "blr_scan_fwd",
    "blr_scan_bwd", "blr_step", "blr_workspace_status", "blr_status_string",
    "blr_selftest_wait_timeout", "blr_scan_fwd_noalloc", "blr_scan_fwd_gated", "blr_scan_bwd_gated",
    "blr_steps", "blr_scan_fwd_varlen", "blr_scan_bwd_varlen", "blr_scan_family",
    "FAMILY_NONE", "FAMILY_TILED", "FAMILY_SERIAL", "FAMILY_SEGMENTED",
    "BDLRUScan", "library_loaded",
]


class BLRError(RuntimeError):
    def __init__(self, status: int, where: str):
        lib = load()
        detail = lib.blr_last_error_string().decode()
        msg = f"{where}: {lib.blr_status_string(status).decode()}"
        if detail:
            msg += f" ({detail})"
        super().__init__(msg)
        self.status = status


def Desc(B: int, L: int, D: int, io: int = BLR_F32, c: float = 1.0) -> blr_desc:
    return blr_desc(B, L, D, io, c)


def library_loaded() -> bool:
    return load() is not None


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.float32:
        return BLR_F32
    if t.dtype == torch.bfloat16:
        return BLR_BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def _ptr(t, name: str):
    """Device pointer of a CUDA tensor on the current device (or a raw int / None)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    import torch
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name}: expected a CUDA tensor, an int pointer or None")
    if t.numel() == 0:
        return None
    if not t.is_cuda or t.device.index != torch.cuda.current_device():
        raise ValueError(f"{name}: tensor must be on the current CUDA device")
    if not t.is_contiguous():
        raise ValueError(f"{name}: tensor must be contiguous")
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status: int, where: str):
    if status != BLR_OK:
        raise BLRError(status, where)


def blr_workspace_bytes(desc: blr_desc) -> int:
    return int(load().blr_workspace_bytes(ctypes.byref(desc)))


# blr_scan_family results
FAMILY_NONE, FAMILY_TILED, FAMILY_SERIAL, FAMILY_SEGMENTED = 0, 1, 2, 3


def blr_scan_family(desc: blr_desc, with_lengths: bool = False) -> int:
    return int(load().blr_scan_family(ctypes.byref(desc), 1 if with_lengths else 0))


def blr_scan_fwd(desc, x, gate_logits, lam, h0, h, h_last, ws, stream=None):
    ws_bytes = ws.numel() if ws is not None and not isinstance(ws, int) else blr_workspace_bytes(desc)
    _check(load().blr_scan_fwd(ctypes.byref(desc), _ptr(x, "x"), _ptr(gate_logits, "gate_logits"),
                               _ptr(lam, "lambda"), _ptr(h0, "h0"), _ptr(h, "h"),
                               _ptr(h_last, "h_last"), _ptr(ws, "ws"), ws_bytes, _stream(stream)),
           "blr_scan_fwd")


def blr_scan_bwd(desc, dh, dh_last, x, gate_logits, lam, h0, dx, dgate_logits, dlam, dh0, ws,
                 stream=None):
    ws_bytes = ws.numel() if ws is not None and not isinstance(ws, int) else blr_workspace_bytes(desc)
    _check(load().blr_scan_bwd(ctypes.byref(desc), _ptr(dh, "dh"), _ptr(dh_last, "dh_last"),
                               _ptr(x, "x"), _ptr(gate_logits, "gate_logits"), _ptr(lam, "lambda"),
                               _ptr(h0, "h0"), _ptr(dx, "dx"), _ptr(dgate_logits, "dgate_logits"),
                               _ptr(dlam, "dlambda"), _ptr(dh0, "dh0"), _ptr(ws, "ws"), ws_bytes,
                               _stream(stream)),
           "blr_scan_bwd")


def blr_scan_fwd_varlen(desc, lengths, x, gate_logits, lam, h0, h, h_last, ws, stream=None):
    """blr_scan_fwd for rows of their own lengths (int32, on the device)."""
    ws_bytes = ws.numel() if ws is not None and not isinstance(ws, int) else blr_workspace_bytes(desc)
    _check(load().blr_scan_fwd_varlen(ctypes.byref(desc), _ptr(lengths, "lengths"), _ptr(x, "x"),
                                      _ptr(gate_logits, "gate_logits"), _ptr(lam, "lambda"),
                                      _ptr(h0, "h0"), _ptr(h, "h"), _ptr(h_last, "h_last"),
                                      _ptr(ws, "ws"), ws_bytes, _stream(stream)),
           "blr_scan_fwd_varlen")


def blr_scan_bwd_varlen(desc, lengths, dh, dh_last, x, gate_logits, lam, h0, dx, dgate_logits,
                        dlam, dh0, ws, stream=None):
    ws_bytes = ws.numel() if ws is not None and not isinstance(ws, int) else blr_workspace_bytes(desc)
    _check(load().blr_scan_bwd_varlen(ctypes.byref(desc), _ptr(lengths, "lengths"), _ptr(dh, "dh"),
                                      _ptr(dh_last, "dh_last"), _ptr(x, "x"),
                                      _ptr(gate_logits, "gate_logits"), _ptr(lam, "lambda"),
                                      _ptr(h0, "h0"), _ptr(dx, "dx"),
                                      _ptr(dgate_logits, "dgate_logits"), _ptr(dlam, "dlambda"),
                                      _ptr(dh0, "dh0"), _ptr(ws, "ws"), ws_bytes, _stream(stream)),
           "blr_scan_bwd_varlen")


def blr_scan_fwd_gated(desc, x, gate_logits, lam, h0, z, y, h_last, ws, stream=None):
    ws_bytes = ws.numel() if ws is not None and not isinstance(ws, int) else blr_workspace_bytes(desc)
    _check(load().blr_scan_fwd_gated(ctypes.byref(desc), _ptr(x, "x"),
                                     _ptr(gate_logits, "gate_logits"), _ptr(lam, "lambda"),
                                     _ptr(h0, "h0"), _ptr(z, "z"), _ptr(y, "y"),
                                     _ptr(h_last, "h_last"), _ptr(ws, "ws"), ws_bytes,
                                     _stream(stream)),
           "blr_scan_fwd_gated")


def blr_scan_bwd_gated(desc, dy, dh_last, x, gate_logits, lam, h0, z, dx, dgate_logits, dz, dlam,
                       dh0, ws, stream=None):
    ws_bytes = ws.numel() if ws is not None and not isinstance(ws, int) else blr_workspace_bytes(desc)
    _check(load().blr_scan_bwd_gated(ctypes.byref(desc), _ptr(dy, "dy"), _ptr(dh_last, "dh_last"),
                                     _ptr(x, "x"), _ptr(gate_logits, "gate_logits"),
                                     _ptr(lam, "lambda"), _ptr(h0, "h0"), _ptr(z, "z"),
                                     _ptr(dx, "dx"), _ptr(dgate_logits, "dgate_logits"),
                                     _ptr(dz, "dz"), _ptr(dlam, "dlambda"), _ptr(dh0, "dh0"),
                                     _ptr(ws, "ws"), ws_bytes, _stream(stream)),
           "blr_scan_bwd_gated")


def blr_step(B, D, io, c, h_prev, x_t, gate_logits_t, lam, h_t, stream=None):
    _check(load().blr_step(B, D, io, c, _ptr(h_prev, "h_prev"), _ptr(x_t, "x_t"),
                           _ptr(gate_logits_t, "gate_logits_t"), _ptr(lam, "lambda"),
                           _ptr(h_t, "h_t"), _stream(stream)),
           "blr_step")


def blr_steps(B, K, D, io, state, c, h_prev, x, gate_logits, lam, h_out, h_seq=None, stream=None):
    """K recurrent steps per row (state dtype `state`, BLR_F32 or BLR_BF16)."""
    _check(load().blr_steps(B, K, D, io, state, c, _ptr(h_prev, "h_prev"), _ptr(x, "x"),
                            _ptr(gate_logits, "gate_logits"), _ptr(lam, "lambda"),
                            _ptr(h_out, "h_out"), _ptr(h_seq, "h_seq"), _stream(stream)),
           "blr_steps")


def blr_workspace_status(desc, ws, stream=None) -> int:
    """Status recorded in the workspace by earlier calls (synchronises the
    stream); ws None reads the library's scratch (backward calls made without a
    workspace)."""
    return int(load().blr_workspace_status(ctypes.byref(desc), _ptr(ws, "ws"),
                                           ws.numel() if ws is not None else 0, _stream(stream)))


def blr_selftest_wait_timeout(desc, ws, timeout_ns: int, stream=None):
    _check(load().blr_selftest_wait_timeout(ctypes.byref(desc), _ptr(ws, "ws"), ws.numel(),
                                            timeout_ns, _stream(stream)),
           "blr_selftest_wait_timeout")


def blr_scan_fwd_noalloc(desc, x, gate_logits, lam, h0, h, h_last, stream=None):
    """blr_scan_fwd on the library's static device scratch, for callers that
    cannot allocate a workspace (see include/blr.h)."""
    _check(load().blr_scan_fwd_noalloc(ctypes.byref(desc), _ptr(x, "x"),
                                       _ptr(gate_logits, "gate_logits"), _ptr(lam, "lambda"),
                                       _ptr(h0, "h0"), _ptr(h, "h"), _ptr(h_last, "h_last"),
                                       _stream(stream)),
           "blr_scan_fwd_noalloc")


def blr_status_string(status: int) -> str:
    return load().blr_status_string(status).decode()


def _autograd():
    import torch

    class BDLRUScan(torch.autograd.Function):
        """h = BD-LRU(x; gate_logits, Lambda, h0) with gradients for all four inputs.

        x (B, L, D), gate_logits (B, L, 2D) in float32 or bfloat16; lam (D,) and
        h0 (B, D) or None in float32. Returns (h, h_last)."""

        @staticmethod
        def forward(ctx, x, gate_logits, lam, h0=None, c: float = 1.0):
            B, L, D = x.shape
            desc = Desc(B, L, D, _dtype_code(x), c)
            ws = torch.empty(max(blr_workspace_bytes(desc), 1), dtype=torch.uint8, device=x.device)
            h = torch.empty_like(x)
            h_last = torch.empty(B, D, dtype=torch.float32, device=x.device)
            blr_scan_fwd(desc, x, gate_logits, lam, h0, h, h_last, ws)
            ctx.save_for_backward(x, gate_logits, lam, h0, ws)
            ctx.desc = desc
            return h, h_last

        @staticmethod
        def backward(ctx, dh, dh_last):
            x, gate_logits, lam, h0, ws = ctx.saved_tensors
            desc = ctx.desc
            B, L, D = x.shape
            dh = torch.zeros_like(x) if dh is None else dh.contiguous()
            dh_last = None if dh_last is None else dh_last.contiguous().float()
            dx = torch.empty_like(x)
            dgl = torch.empty_like(gate_logits)
            dlam = torch.empty(D, dtype=torch.float32, device=x.device)
            dh0 = torch.empty(B, D, dtype=torch.float32, device=x.device) if h0 is not None else None
            blr_scan_bwd(desc, dh, dh_last, x, gate_logits, lam, h0, dx, dgl, dlam, dh0, ws)
            return dx, dgl, dlam, dh0, None

    return BDLRUScan


def __getattr__(name):
    if name == "BDLRUScan":
        cls = _autograd()
        globals()["BDLRUScan"] = cls
        return cls
    raise AttributeError(name)
