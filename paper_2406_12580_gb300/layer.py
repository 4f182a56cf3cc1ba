"""The gated recurrent layer of RecBLR (Alg. 1) around the library's kernels.

    H_x, H_z = Linear(H_i), Linear(H_i)            expand D -> E D (one GEMM, two halves)
    H'_x     = SiLU(Conv1d(H_x))                   causal, depthwise along time
    rho|iota = Linear(H'_x)                        the gate logits (Sec. 3.2, W_r x + b_r, W_i x + b_i)
    H'_y     = BD-LRU(H'_x) * SiLU(H_z)            blr_scan_fwd_gated: the scan and the merge, fused
    H_o      = Linear(H'_y)                        reduce E D -> D

The GEMMs and the convolution are torch operators (cuBLAS, cuDNN); the scan and
the merge, forward and backward, run in the library (``BDLRUGatedScan``). The
decay parameter Lambda is initialised as in Sec. 3.2: exp(-softplus(Lambda))
uniform in [0.9, 0.999]. The convolution width is not given in the paper; it
is a parameter (default 4).
"""
from __future__ import annotations

import torch
from torch import nn

from . import (Desc, _dtype_code, blr_scan_bwd_gated, blr_scan_fwd_gated, blr_workspace_bytes)


class BDLRUGatedScan(torch.autograd.Function):
    """y = BD-LRU(x; gate_logits, Lambda, h0) * SiLU(z), with gradients for x,
    gate_logits, Lambda, z and h0. x, z (B, L, D) and gate_logits (B, L, 2D) in
    float32 or bfloat16; lam (D,) and h0 (B, D) or None in float32. Returns
    (y, h_last)."""

    @staticmethod
    def forward(ctx, x, gate_logits, lam, z, h0=None, c: float = 1.0):
        B, L, D = x.shape
        x, gate_logits, z = x.contiguous(), gate_logits.contiguous(), z.contiguous()
        ctx.lam_dtype = lam.dtype
        lam = lam.contiguous().float()
        desc = Desc(B, L, D, _dtype_code(x), c)
        ws = torch.empty(max(blr_workspace_bytes(desc), 16), dtype=torch.uint8, device=x.device)
        y = torch.empty_like(x)
        h_last = torch.empty(B, D, dtype=torch.float32, device=x.device)
        blr_scan_fwd_gated(desc, x, gate_logits, lam, h0, z, y, h_last, ws)
        ctx.save_for_backward(x, gate_logits, lam, z, h0, ws)
        ctx.desc = desc
        return y, h_last

    @staticmethod
    def backward(ctx, dy, dh_last):
        x, gate_logits, lam, z, h0, ws = ctx.saved_tensors
        B, L, D = x.shape
        dy = torch.zeros_like(x) if dy is None else dy.contiguous().to(x.dtype)
        dh_last = None if dh_last is None else dh_last.contiguous().float()
        dx = torch.empty_like(x)
        dgl = torch.empty_like(gate_logits)
        dz = torch.empty_like(z)
        dlam = torch.empty(D, dtype=torch.float32, device=x.device)
        dh0 = torch.empty(B, D, dtype=torch.float32, device=x.device) if h0 is not None else None
        blr_scan_bwd_gated(ctx.desc, dy, dh_last, x, gate_logits, lam, h0, z, dx, dgl, dz, dlam,
                           dh0, ws)
        return dx, dgl, dlam.to(ctx.lam_dtype), dz, dh0, None


def lambda_init(n: int, lo: float = 0.9, hi: float = 0.999, generator=None) -> torch.Tensor:
    """Lambda with exp(-softplus(Lambda)) ~ U[lo, hi] (Sec. 3.2)."""
    u = torch.rand(n, generator=generator, dtype=torch.float64) * (hi - lo) + lo
    return torch.log((1.0 - u) / u).float()


class GatedRecurrentLayer(nn.Module):
    """Alg. 1 with the BD-LRU and the merge on the library's fused kernels."""

    def __init__(self, d_model: int, expand: int = 2, conv_width: int = 4, c: float = 1.0,
                 device=None, dtype=None):
        super().__init__()
        ed = expand * d_model
        if ed % 8 != 0:
            raise ValueError("expand * d_model must be a multiple of 8")
        kw = dict(device=device, dtype=dtype)
        self.ed, self.c = ed, c
        self.in_proj = nn.Linear(d_model, 2 * ed, **kw)         # H_x | H_z
        self.conv = nn.Conv1d(ed, ed, conv_width, groups=ed, padding=conv_width - 1, **kw)
        self.gate_proj = nn.Linear(ed, 2 * ed, **kw)            # rho | iota
        self.out_proj = nn.Linear(ed, d_model, **kw)
        self.lam = nn.Parameter(lambda_init(ed).to(device=device))

    def forward(self, h: torch.Tensor) -> torch.Tensor:
        B, L, _ = h.shape
        hx, hz = self.in_proj(h).split(self.ed, dim=-1)
        xc = self.conv(hx.transpose(1, 2))[..., :L].transpose(1, 2)   # causal: drop the tail
        x = nn.functional.silu(xc).contiguous()
        gl = self.gate_proj(x).contiguous()
        y, _ = BDLRUGatedScan.apply(x, gl, self.lam, hz.contiguous(), None, self.c)
        return self.out_proj(y)


__all__ = ["BDLRUGatedScan", "GatedRecurrentLayer", "lambda_init"]
