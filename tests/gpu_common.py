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
# Elementwise bounds on max |gpu - oracle| / (|oracle| + 1e-3 max|oracle|)
# (relative per element, absolute below a thousandth of the tensor's scale):
# measured at most 3.2e-4 (float32) and 6e-3 (bfloat16: one output rounding of
# up to 2^-8 relative, plus tanh.approx's 2^-11 in the gates) over the whole
# suite, the long-sequence workload on every channel included.
ELEM_TOL = {I.F32: 2e-3, I.BF16: 2e-2}
# dLambda per channel: |gpu - oracle| / (|oracle| + 1e-6 max|oracle|), so that
# a channel with a small gradient is checked at its own size; measured at most
# 4.1e-4 (float32) and 3.5e-2 (bfloat16, whose per-step terms carry the
# gates' 2^-11 and cancel in the sum over steps).
DLAM_TOL = {I.F32: 4e-3, I.BF16: 0.15}


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


def per_channel(got, want, floor_frac=1e-6) -> float:
    """max |gpu - oracle| / (|oracle| + floor_frac max|oracle|) over a vector."""
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    if want.size == 0:
        return 0.0
    floor = floor_frac * np.max(np.abs(want))
    return float(np.max(np.abs(got - want) / (np.abs(want) + floor))) if floor > 0 else float(
        np.max(np.abs(got - want)))


def elementwise_applies(cfg) -> bool:
    """Whether the elementwise bounds apply: not to the gated layer in
    bfloat16 on the tiled kernels, which compose the merge around the scan and
    round dh = dy SiLU(z) to bfloat16 between kernels, so that gradients that
    nearly cancel lose their relative accuracy there (the normwise bound holds)."""
    if not (cfg.gated and cfg.io == I.BF16):
        return True
    from paper_2406_12580_gb300 import FAMILY_TILED, Desc, blr_scan_family
    return blr_scan_family(Desc(cfg.B, cfg.L, cfg.D, 1, cfg.c)) != FAMILY_TILED


def compare(inp: I.ScanInputs, got: dict, want: dict, tol=None):
    """Asserts the normwise error of every output and, where they apply, the
    elementwise bounds (dLambda per channel); returns {name: (normwise,
    elementwise)}."""
    tol = TOL[inp.cfg.io] if tol is None else tol
    errs = {}
    for k, w in want.items():
        errs[k] = normwise(got[k], w)
    bad = {k: v for k, v in errs.items() if not v <= tol}
    assert not bad, f"{inp.cfg.name}: normwise errors above {tol}: {bad} (all: {errs})"
    out = {k: (v, elementwise(got[k], want[k])) for k, v in errs.items()}
    if tol == TOL[inp.cfg.io] and elementwise_applies(inp.cfg):
        etol = ELEM_TOL[inp.cfg.io]
        bad = {k: e for k, (_, e) in out.items() if not e <= etol}
        assert not bad, f"{inp.cfg.name}: elementwise errors above {etol}: {bad}"
        if want.get("dlam") is not None:
            pc = per_channel(got["dlam"], want["dlam"])
            assert pc <= DLAM_TOL[inp.cfg.io], f"{inp.cfg.name}: dlambda per channel {pc}"
    return out


def compare_by_rows(inp: I.ScanInputs, buf, rows: int = 1, threads: int = 0):
    """A full-size workload against the oracle on every channel, `rows` batch
    rows at a time (the recurrence is independent per batch row and channel;
    dLambda, a sum over rows, is summed over the chunks). The elementwise floor
    is a thousandth of each chunk's largest value."""
    orc = oracle.load()
    cfg = inp.cfg
    names = {"h": "h", "h_last": "h_last", "dx": "dx", "dgl": "dgl", "dh0": "dh0"}
    err, scale, ew = {}, {}, {}
    dlam = None
    for b0 in range(0, cfg.B, rows):
        sl = slice(b0, min(cfg.B, b0 + rows))
        pick = lambda a: None if a is None else np.ascontiguousarray(a[sl])  # noqa: E731
        h, h_last = orc.fwd(pick(inp.x), pick(inp.gl), inp.lam, pick(inp.h0), c=cfg.c,
                            threads=threads)
        want = {"h": h, "h_last": h_last}
        if inp.dh is not None:
            dx, dgl, dl, dh0 = orc.bwd(pick(inp.dh), pick(inp.x), pick(inp.gl), inp.lam,
                                       pick(inp.h0), pick(inp.dh_last), c=cfg.c, threads=threads)
            want.update(dx=dx, dgl=dgl, dh0=dh0)
            dlam = dl if dlam is None else dlam + dl
        for k, w in want.items():
            g = to_host_f64(getattr(buf, names[k])[sl])
            err[k] = max(err.get(k, 0.0), float(np.max(np.abs(g - w))))
            scale[k] = max(scale.get(k, 0.0), float(np.max(np.abs(w))))
            ew[k] = max(ew.get(k, 0.0), elementwise(g, w))
    out = {k: (err[k] / scale[k] if scale[k] > 0 else err[k], ew[k]) for k in err}
    if dlam is not None:
        g = to_host_f64(buf.dlam)
        out["dlam"] = (normwise(g, dlam), elementwise(g, dlam))
        pc = per_channel(g, dlam)
        assert pc <= DLAM_TOL[cfg.io], f"{cfg.name}: dlambda per channel {pc}"
    tol, etol = TOL[cfg.io], ELEM_TOL[cfg.io]
    bad = {k: v for k, v in out.items() if not (v[0] <= tol and v[1] <= etol)}
    assert not bad, f"{cfg.name}: errors above ({tol}, {etol}): {bad}"
    return out


def gpu_step(sinp: I.StepInputs):
    import torch
    buf = StepBuffers.from_inputs(sinp)
    buf.step()
    torch.cuda.synchronize()
    return buf
