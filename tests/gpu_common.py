"""Shared helpers of the GPU parity tests: run the CUDA path through the C ABI
and the float64 oracle on the same seeded inputs, and compare them."""
from __future__ import annotations

import numpy as np

import oracle
from paper_2406_12580_gb300 import inputs as I
from paper_2406_12580_gb300.device import ScanBuffers, StepBuffers, to_host_f64

# Tolerances on the normwise relative error max|gpu - oracle| / max|oracle|:
# 1e-5 for float32 I/O and 2e-2 for bfloat16 I/O (bf16 outputs alone carry a
# relative rounding error of up to 2^-9 = 2e-3).
TOL = {I.F32: 1e-5, I.BF16: 2e-2}


def normwise(got, want) -> float:
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    assert got.shape == want.shape, (got.shape, want.shape)
    if want.size == 0:
        return 0.0
    scale = np.max(np.abs(want))
    err = np.max(np.abs(got - want))
    if scale == 0.0:
        return float(err)
    return float(err / scale)


def gpu_scan(inp: I.ScanInputs, with_bwd=True, sync=True):
    import torch
    buf = ScanBuffers.from_inputs(inp, with_bwd=with_bwd)
    buf.fwd()
    if with_bwd and buf.dh is not None:
        buf.bwd()
    if sync:
        torch.cuda.synchronize()
    return buf


def gpu_scan_gated(inp: I.ScanInputs, with_bwd=True):
    """The gated entry points (y = h SiLU(z) in buf.h; dz in buf.dz)."""
    import torch
    buf = ScanBuffers.from_inputs(inp, with_bwd=with_bwd)
    buf.fwd_gated()
    if with_bwd and buf.dh is not None:
        buf.bwd_gated()
    torch.cuda.synchronize()
    return buf


def gpu_outputs(buf, dsel=None):
    """Outputs as float64 numpy arrays, optionally only the channels `dsel`."""
    import torch
    out = {}
    D = buf.desc.D

    def take(t, chan_axis_size):
        if t is None:
            return None
        if dsel is None:
            return to_host_f64(t)
        idx = torch.as_tensor(dsel, device=t.device)
        if chan_axis_size == 2 * D:
            idx = torch.cat([idx, idx + D])
        return to_host_f64(t.index_select(t.dim() - 1, idx))

    out["h"] = take(buf.h, D)
    out["h_last"] = take(buf.h_last, D)
    if buf.dx is not None:
        out["dx"] = take(buf.dx, D)
        out["dgl"] = take(buf.dgl, 2 * D)
        out["dlam"] = take(buf.dlam, D)
        out["dh0"] = take(buf.dh0, D)
    if buf.dz is not None:
        out["dz"] = take(buf.dz, D)
    return out


def select_channels(inp: I.ScanInputs, dsel):
    """The inputs restricted to channels `dsel` (the recurrence is per channel)."""
    D = inp.cfg.D
    dsel = np.asarray(dsel)
    gidx = np.concatenate([dsel, dsel + D])
    pick = lambda a, ax_idx: None if a is None else np.ascontiguousarray(a[..., ax_idx])  # noqa: E731
    return dict(x=pick(inp.x, dsel), gl=pick(inp.gl, gidx), lam=inp.lam[dsel],
                h0=pick(inp.h0, dsel), dh=pick(inp.dh, dsel), dh_last=pick(inp.dh_last, dsel),
                z=pick(inp.z, dsel))


def oracle_outputs(inp: I.ScanInputs, dsel=None, threads=0):
    orc = oracle.load()
    cfg = inp.cfg
    if dsel is None:
        a = dict(x=inp.x, gl=inp.gl, lam=inp.lam, h0=inp.h0, dh=inp.dh, dh_last=inp.dh_last,
                 z=inp.z)
    else:
        a = select_channels(inp, dsel)
    if a["z"] is not None:  # the gated layer: h holds y = h SiLU(z), dh is dy
        y, h_last = orc.fwd_gated(a["x"], a["gl"], a["lam"], a["z"], a["h0"], c=cfg.c,
                                  threads=threads)
        out = {"h": y, "h_last": h_last}
        if a["dh"] is not None:
            dx, dgl, dlam, dh0, dz = orc.bwd_gated(a["dh"], a["x"], a["gl"], a["lam"], a["z"],
                                                   a["h0"], a["dh_last"], c=cfg.c, threads=threads)
            out.update(dx=dx, dgl=dgl, dlam=dlam, dh0=dh0, dz=dz)
        return out
    h, h_last = orc.fwd(a["x"], a["gl"], a["lam"], a["h0"], c=cfg.c, threads=threads)
    out = {"h": h, "h_last": h_last}
    if a["dh"] is not None:
        dx, dgl, dlam, dh0 = orc.bwd(a["dh"], a["x"], a["gl"], a["lam"], a["h0"], a["dh_last"],
                                     c=cfg.c, threads=threads)
        out.update(dx=dx, dgl=dgl, dlam=dlam, dh0=dh0)
    return out


def elementwise(got, want) -> float:
    """Diagnostic beside the normwise error: max |gpu - oracle| / (|oracle| +
    1e-3 max|oracle|), relative per element but defined at exact zeros."""
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    if want.size == 0:
        return 0.0
    floor = 1e-3 * np.max(np.abs(want))
    if floor == 0.0:
        return float(np.max(np.abs(got - want)))
    return float(np.max(np.abs(got - want) / (np.abs(want) + floor)))


def compare(inp: I.ScanInputs, got: dict, want: dict, tol=None):
    """Asserts the normwise error of every output; returns it with the
    elementwise diagnostic ({name: (normwise, elementwise)})."""
    tol = TOL[inp.cfg.io] if tol is None else tol
    errs = {}
    for k, w in want.items():
        errs[k] = normwise(got[k], w)
    bad = {k: v for k, v in errs.items() if not v <= tol}
    assert not bad, f"{inp.cfg.name}: normwise errors above {tol}: {bad} (all: {errs})"
    return {k: (v, elementwise(got[k], want[k])) for k, v in errs.items()}


def gpu_step(sinp: I.StepInputs):
    import torch
    buf = StepBuffers.from_inputs(sinp)
    buf.step()
    torch.cuda.synchronize()
    return buf
