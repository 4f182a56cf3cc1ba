"""Device buffers for one scan problem (torch is used for memory and streams only).

``ScanBuffers`` holds the inputs of a synthetic workload on the GPU, the
outputs of the forward and backward, and the workspace, and runs the C-ABI
calls on them. Nothing here computes any part of the method.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import numpy as np

from . import (BLR_BF16, BLR_F32, Desc, blr_scan_bwd, blr_scan_bwd_gated, blr_scan_bwd_varlen,
               blr_scan_fwd, blr_scan_fwd_gated, blr_scan_fwd_varlen, blr_step, blr_workspace_bytes)
from .inputs import BF16, ScanInputs, StepInputs


def torch_io_dtype(io: str):
    import torch
    return torch.bfloat16 if io == BF16 else torch.float32


def io_code(io: str) -> int:
    return BLR_BF16 if io == BF16 else BLR_F32


def to_device(a: Optional[np.ndarray], io: str, device, pin: bool = False):
    """Upload a generator array: float32 values, or uint16 bf16 bit patterns."""
    import torch
    if a is None:
        return None
    if a.dtype == np.uint16:
        t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    if pin:
        t = t.pin_memory()
    return t.to(device, non_blocking=pin)


def to_host_f64(t) -> Optional[np.ndarray]:
    if t is None:
        return None
    return t.detach().float().cpu().numpy().astype(np.float64)


@dataclass
class ScanBuffers:
    desc: object
    x: object
    gl: object
    lam: object
    h0: object
    dh: object
    dh_last: object
    h: object
    h_last: object
    dx: object
    dgl: object
    dlam: object
    dh0: object
    ws: object
    z: object = None   # gated workloads: the merge's input (then h holds y and dh is dy)
    dz: object = None

    @classmethod
    def from_inputs(cls, inp: ScanInputs, device="cuda", with_bwd: bool = True):
        import torch
        cfg = inp.cfg
        B, L, D = cfg.B, cfg.L, cfg.D
        io_t = torch_io_dtype(cfg.io)
        desc = Desc(B, L, D, io_code(cfg.io), cfg.c)
        f32 = torch.float32
        up = lambda name: to_device(inp.io_array(name), cfg.io, device)  # noqa: E731
        x, gl = up("x"), up("gl")
        lam = to_device(inp.lam, "f32", device)
        h0 = to_device(inp.h0, "f32", device)
        dh = up("dh") if (with_bwd and inp.dh is not None) else None
        dh_last = to_device(inp.dh_last, "f32", device) if with_bwd else None
        ws = torch.empty(max(blr_workspace_bytes(desc), 16), dtype=torch.uint8, device=device)
        h = torch.empty(B, L, D, dtype=io_t, device=device)
        h_last = torch.empty(B, D, dtype=f32, device=device)
        bwd = with_bwd and dh is not None
        dx = torch.empty(B, L, D, dtype=io_t, device=device) if bwd else None
        dgl = torch.empty(B, L, 2 * D, dtype=io_t, device=device) if bwd else None
        dlam = torch.empty(D, dtype=f32, device=device) if bwd else None
        dh0 = torch.empty(B, D, dtype=f32, device=device) if bwd else None
        z = up("z") if inp.z is not None else None
        dz = torch.empty(B, L, D, dtype=io_t, device=device) if (bwd and z is not None) else None
        return cls(desc, x, gl, lam, h0, dh, dh_last, h, h_last, dx, dgl, dlam, dh0, ws, z, dz)

    def fwd(self, stream=None, write_h: bool = True):
        blr_scan_fwd(self.desc, self.x, self.gl, self.lam, self.h0, self.h if write_h else None,
                     self.h_last, self.ws, stream)

    def bwd(self, stream=None):
        blr_scan_bwd(self.desc, self.dh, self.dh_last, self.x, self.gl, self.lam, self.h0, self.dx,
                     self.dgl, self.dlam, self.dh0, self.ws, stream)

    def fwd_varlen(self, lengths, stream=None):
        """The forward with per-row lengths (an int32 CUDA tensor of B)."""
        blr_scan_fwd_varlen(self.desc, lengths, self.x, self.gl, self.lam, self.h0, self.h,
                            self.h_last, self.ws, stream)

    def bwd_varlen(self, lengths, stream=None):
        blr_scan_bwd_varlen(self.desc, lengths, self.dh, self.dh_last, self.x, self.gl, self.lam,
                            self.h0, self.dx, self.dgl, self.dlam, self.dh0, self.ws, stream)

    def fwd_gated(self, stream=None):
        """y = h SiLU(z) into self.h."""
        blr_scan_fwd_gated(self.desc, self.x, self.gl, self.lam, self.h0, self.z, self.h,
                           self.h_last, self.ws, stream)

    def bwd_gated(self, stream=None):
        """Backward of fwd_gated with self.dh as dy."""
        blr_scan_bwd_gated(self.desc, self.dh, self.dh_last, self.x, self.gl, self.lam, self.h0,
                           self.z, self.dx, self.dgl, self.dz, self.dlam, self.dh0, self.ws, stream)


@dataclass
class StepBuffers:
    B: int
    D: int
    io: int
    c: float
    h_prev: object
    x: object
    gl: object
    lam: object
    h_t: object

    @classmethod
    def from_inputs(cls, inp: StepInputs, device="cuda"):
        import torch
        cfg = inp.cfg
        up = lambda name: to_device(inp.io_array(name), cfg.io, device)  # noqa: E731
        h_prev = to_device(inp.h_prev, "f32", device)
        return cls(cfg.B, cfg.D, io_code(cfg.io), cfg.c, h_prev, up("x"), up("gl"),
                   to_device(inp.lam, "f32", device),
                   torch.empty(cfg.B, cfg.D, dtype=torch.float32, device=device))

    def step(self, stream=None):
        blr_step(self.B, self.D, self.io, self.c, self.h_prev, self.x, self.gl, self.lam, self.h_t,
                 stream)
