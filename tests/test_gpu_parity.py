"""GPU: the CUDA path (through the C ABI) against the float64 oracle.

Every comparison uses the same seeded inputs on both sides (bf16 inputs are
rounded once by the generator; the oracle upcasts them). Errors are normwise:
max|gpu - oracle| / max|oracle| <= 1e-5 for float32 I/O and <= 2e-2 for
bfloat16 I/O.
"""
import numpy as np
import pytest

from gpu_common import (TOL, compare, compare_by_rows, gpu_outputs, gpu_scan, gpu_scan_gated,
                        gpu_step, normwise, oracle_outputs)
from paper_2406_12580_gb300 import inputs as I

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, but never run there
    pytest.skip("no CUDA device", allow_module_level=True)

# Small and ragged shapes the oracle runs in full: a single element, one and
# several partial tiles, a partial channel block (D = 72 = 64 + 8), the
# minimal channel width, long look-back chains, slow decays, random h0 and
# dh_last, and c != 1.
SMALL = [
    dict(B=1, L=1, D=8),
    dict(B=2, L=3, D=8, random_h0=True, random_dh_last=True),
    dict(B=3, L=7, D=16),
    dict(B=4, L=50, D=64),
    dict(B=3, L=65, D=72, random_h0=True, random_dh_last=True),
    dict(B=2, L=300, D=16, random_h0=True),
    dict(B=1, L=4000, D=8, random_dh_last=True),
    dict(B=2, L=1031, D=256, decay=(0.99, 0.9999), random_h0=True, random_dh_last=True),
    dict(B=5, L=129, D=128, c=2.5, random_h0=True),
    dict(B=2, L=200, D=64, gate_std=3.0, x_std=4.0),
    # enough (batch row, channel group) chains for the serial kernels, with
    # partial channel groups and sequence tails
    dict(B=2100, L=5, D=32, random_h0=True, random_dh_last=True),
    dict(B=700, L=37, D=40, random_h0=True),
    dict(B=1100, L=130, D=16, random_dh_last=True, decay=(0.99, 0.9999)),
    # serial chains split into time segments (2 or 4 warps per chain), with a
    # short last segment, h0 and dh_last entering through the segment maps
    dict(B=300, L=203, D=24, random_h0=True, random_dh_last=True),
    dict(B=600, L=100, D=72, random_h0=True, random_dh_last=True),
    dict(B=520, L=129, D=32, decay=(0.99, 0.9999)),
    # fast decays (exp(-softplus(Lambda)) down to 0.05, so |log alpha| > 0.25:
    # the general e^l - 1 branch) and c != 1, on the serial and tiled families
    dict(B=3, L=150, D=40, decay=(0.05, 0.95), c=3.0, random_h0=True, random_dh_last=True),
    dict(B=400, L=90, D=40, decay=(0.05, 0.95), c=0.5, random_h0=True, random_dh_last=True),
    # a long sequence with many chains (float32: the forward's 32-row boxes),
    # ending in a partial box
    dict(B=260, L=1100, D=8, decay=(0.99, 0.9999), random_h0=True, random_dh_last=True),
]


def _cfg(io, seed, **kw):
    return I.ScanConfig(f"small {kw} {io}", io=io, seed=seed, **kw)


@pytest.mark.parametrize("io", [I.F32, I.BF16])
@pytest.mark.parametrize("case", range(len(SMALL)))
def test_small_shapes(io, case):
    inp = I.make_scan_inputs(_cfg(io, 100 + case, **SMALL[case]))
    buf = gpu_scan(inp)
    compare(inp, gpu_outputs(buf), oracle_outputs(inp))


@pytest.mark.parametrize("k", [0, 1, 2])
def test_config_full_oracle(k):
    """Configurations 0-2 at full size against the full oracle."""
    inp = I.make_scan_inputs(I.CONFIGS[k])
    buf = gpu_scan(inp)
    errs = compare(inp, gpu_outputs(buf), oracle_outputs(inp, threads=0))
    print(f"config {k}: {errs}")


def _sampled_channels(D):
    return sorted({0, 1, 7, 8, 63, 64, 65, D // 2, D - 9, D - 1} & set(range(D)))


@pytest.mark.parametrize("k", [3, 4])
def test_config_full_size_every_channel(k):
    """Configurations 3-4 at full size against the oracle on every batch row
    and channel, a few batch rows at a time (which bounds host memory)."""
    inp = I.make_scan_inputs(I.CONFIGS[k])
    buf = gpu_scan(inp)
    errs = compare_by_rows(inp, buf, rows=1 if k == 4 else 8)
    print(f"config {k}: {errs}")


@pytest.mark.parametrize("io", [I.F32, I.BF16])
def test_step_full(io):
    cfg = I.StepConfig(f"step {io}", B=65536, D=64, io=io, seed=4)
    s = I.make_step_inputs(cfg)
    buf = gpu_step(s)
    import oracle
    want = oracle.load().step(s.h_prev, s.x, s.gl, s.lam, c=cfg.c)
    got = buf.h_t.cpu().numpy().astype(np.float64)
    # the state is float32 in both dtypes; bf16 only rounds the inputs, which
    # both sides share, and the fast gate arithmetic stays near 1e-6
    assert normwise(got, want) <= (1e-5 if io == I.F32 else 1e-4)


def test_step_small_and_aliased():
    cfg = I.StepConfig("step small", B=3, D=24, io=I.F32, seed=9)
    s = I.make_step_inputs(cfg)
    import oracle
    want = oracle.load().step(s.h_prev, s.x, s.gl, s.lam)
    from paper_2406_12580_gb300 import BLR_F32, blr_step
    from paper_2406_12580_gb300.device import to_device
    h = to_device(s.h_prev, "f32", "cuda")
    x = to_device(s.x, "f32", "cuda")
    gl = to_device(s.gl, "f32", "cuda")
    lam = to_device(s.lam, "f32", "cuda")
    blr_step(3, 24, BLR_F32, 1.0, h, x, gl, lam, h)  # in place: h_t aliases h_prev
    torch.cuda.synchronize()
    assert normwise(h.cpu().numpy(), want) <= 1e-5


def test_padding_rows_are_exact_zeros():
    """Config 2's left-padded rows (x = rho = iota = 0, h0 = 0) stay exactly 0
    (the embedding-padding claim of Sec. 3.3), and diota vanishes there."""
    inp = I.make_scan_inputs(I.scaled(I.CONFIGS[2], B=256))
    buf = gpu_scan(inp)
    p = inp.cfg.pad_rows
    assert torch.count_nonzero(buf.h[:, :p]).item() == 0
    assert torch.count_nonzero(buf.dgl[:, :p, inp.cfg.D:]).item() == 0
    # and the real rows equal a run without the padding
    cfg2 = I.scaled(inp.cfg, L=inp.cfg.L - p, pad_frac=0.0)
    inp2 = I.make_scan_inputs(cfg2)
    inp2.x, inp2.gl = inp.x[:, p:].copy(), inp.gl[:, p:].copy()
    inp2.bits = {k: np.ascontiguousarray(v[:, p:]) for k, v in inp.bits.items()}
    inp2.dh = inp.dh[:, p:].copy()
    buf2 = gpu_scan(inp2, with_bwd=False)
    # chunk boundaries move with the padding, so float32 rounding may differ
    assert normwise(buf.h[:, p:].float().cpu().numpy(), buf2.h.float().cpu().numpy()) <= 1e-2


def test_split_resume():
    cfg = I.ScanConfig("split", B=3, L=500, D=64, io=I.F32, seed=31, random_h0=True)
    inp = I.make_scan_inputs(cfg)
    full = gpu_scan(inp, with_bwd=False)
    k = 217
    a = I.make_scan_inputs(I.scaled(cfg, L=k))
    a.x, a.gl, a.h0 = inp.x[:, :k].copy(), inp.gl[:, :k].copy(), inp.h0
    ba = gpu_scan(a, with_bwd=False)
    b = I.make_scan_inputs(I.scaled(cfg, L=cfg.L - k))
    b.x, b.gl, b.h0 = inp.x[:, k:].copy(), inp.gl[:, k:].copy(), ba.h_last.cpu().numpy()
    bb = gpu_scan(b, with_bwd=False)
    got = torch.cat([ba.h, bb.h], dim=1).cpu().numpy()
    assert normwise(got, full.h.cpu().numpy()) <= 1e-6
    assert normwise(bb.h_last.cpu().numpy(), full.h_last.cpu().numpy()) <= 1e-6


def test_carries_only_forward_then_backward():
    cfg = I.ScanConfig("carries", B=4, L=700, D=64, io=I.F32, seed=32, random_h0=True,
                       random_dh_last=True)
    inp = I.make_scan_inputs(cfg)
    from paper_2406_12580_gb300.device import ScanBuffers
    buf = ScanBuffers.from_inputs(inp)
    buf.h.fill_(7.0)
    buf.fwd(write_h=False)
    buf.bwd()
    torch.cuda.synchronize()
    assert torch.all(buf.h == 7.0)  # h untouched
    want = oracle_outputs(inp)
    got = gpu_outputs(buf)
    for k in ("h_last", "dx", "dgl", "dlam", "dh0"):
        assert normwise(got[k], want[k]) <= TOL[I.F32], k
    # the backward can be repeated on the same workspace
    buf.bwd()
    torch.cuda.synchronize()
    got2 = gpu_outputs(buf)
    for k in ("dx", "dgl", "dlam", "dh0"):
        assert normwise(got2[k], want[k]) <= TOL[I.F32], k


def test_empty_sequence_and_batch():
    from paper_2406_12580_gb300 import Desc, blr_scan_bwd, blr_scan_fwd
    B, D = 3, 16
    h0 = torch.randn(B, D, device="cuda")
    dh_last = torch.randn(B, D, device="cuda")
    lam = torch.randn(D, device="cuda")
    h_last = torch.full((B, D), 5.0, device="cuda")
    e = torch.empty(0, device="cuda")
    blr_scan_fwd(Desc(B, 0, D), e, e, lam, h0, e, h_last, None)
    dlam = torch.full((D,), 5.0, device="cuda")
    dh0 = torch.full((B, D), 5.0, device="cuda")
    blr_scan_bwd(Desc(B, 0, D), e, dh_last, e, e, lam, h0, e, e, dlam, dh0, None)
    torch.cuda.synchronize()
    assert torch.equal(h_last, h0) and torch.equal(dh0, dh_last)
    assert torch.count_nonzero(dlam).item() == 0
    blr_scan_fwd(Desc(B, 0, D), e, e, lam, None, e, h_last, None)
    blr_scan_bwd(Desc(B, 0, D), e, None, e, e, lam, None, e, e, dlam, dh0, None)
    torch.cuda.synchronize()
    assert torch.count_nonzero(h_last).item() == 0 and torch.count_nonzero(dh0).item() == 0
    blr_scan_fwd(Desc(0, 10, D), e, e, lam, None, e, None, None)  # B = 0: nothing to do


def test_chained_optional_arguments():
    """The chained kernels (one long bfloat16 row) with every optional pointer
    NULL: no h0, h, h_last in the forward (carries only), no dh_last and dh0
    in the backward; then the backward again on the same workspace, which
    must give the same gradients (its records are emptied again each call)."""
    from paper_2406_12580_gb300 import (FAMILY_SEGMENTED, Desc, blr_scan_bwd, blr_scan_family,
                                        blr_scan_fwd)
    from paper_2406_12580_gb300.device import ScanBuffers
    cfg = I.ScanConfig("chained, optional arguments NULL", B=1, L=16500, D=72, io=I.BF16, seed=35)
    desc = Desc(cfg.B, cfg.L, cfg.D, 1, cfg.c)
    assert blr_scan_family(desc) == FAMILY_SEGMENTED
    inp = I.make_scan_inputs(cfg)
    assert inp.h0 is None and inp.dh_last is None
    buf = ScanBuffers.from_inputs(inp)
    buf.h.fill_(7.0)
    blr_scan_fwd(buf.desc, buf.x, buf.gl, buf.lam, None, None, None, buf.ws)
    blr_scan_bwd(buf.desc, buf.dh, None, buf.x, buf.gl, buf.lam, None, buf.dx, buf.dgl, buf.dlam,
                 None, buf.ws)
    torch.cuda.synchronize()
    assert torch.all(buf.h == 7.0)  # h untouched
    want = oracle_outputs(inp)
    got = gpu_outputs(buf)
    compare(inp, {k: got[k] for k in ("dx", "dgl", "dlam")},
            {k: want[k] for k in ("dx", "dgl", "dlam")})
    first = [buf.dx.clone(), buf.dgl.clone(), buf.dlam.clone()]
    blr_scan_bwd(buf.desc, buf.dh, None, buf.x, buf.gl, buf.lam, None, buf.dx, buf.dgl, buf.dlam,
                 None, buf.ws)
    torch.cuda.synchronize()
    # the look-back folds whichever predecessors have published, so a repeat may
    # differ from the first call by one bfloat16 unit in the last place
    for a, b in zip(first, [buf.dx, buf.dgl, buf.dlam]):
        assert normwise(b.float().cpu().numpy(), a.float().cpu().numpy()) <= 2.0 ** -7


def test_backward_without_forward_carries_is_reported():
    from paper_2406_12580_gb300 import (BLR_ERR_WORKSPACE, BLR_OK, Desc, blr_workspace_status)
    from paper_2406_12580_gb300.device import ScanBuffers
    cfg = I.ScanConfig("ws", B=2, L=300, D=64, io=I.F32, seed=33)
    inp = I.make_scan_inputs(cfg)
    buf = ScanBuffers.from_inputs(inp)
    buf.ws.zero_()
    buf.dx.fill_(3.0)
    buf.bwd()
    assert blr_workspace_status(buf.desc, buf.ws) == BLR_ERR_WORKSPACE
    assert torch.all(buf.dx == 3.0)
    buf.fwd()  # a forward clears the error word and fills the carries
    buf.bwd()
    assert blr_workspace_status(buf.desc, buf.ws) == BLR_OK
    # a forward of another length leaves carries that do not match this problem
    other = Desc(2, 299, 64)
    from paper_2406_12580_gb300 import blr_scan_fwd
    blr_scan_fwd(other, buf.x, buf.gl, buf.lam, None, None, None, buf.ws)
    buf.bwd()
    assert blr_workspace_status(buf.desc, buf.ws) == BLR_ERR_WORKSPACE


def test_bounded_wait_reports_timeout():
    from paper_2406_12580_gb300 import (BLR_ERR_TIMEOUT, BLR_OK, blr_selftest_wait_timeout,
                                        blr_workspace_status)
    from paper_2406_12580_gb300.device import ScanBuffers
    inp = I.make_scan_inputs(I.ScanConfig("timeout", B=2, L=100, D=64, io=I.F32, seed=34))
    buf = ScanBuffers.from_inputs(inp)
    buf.fwd()
    assert blr_workspace_status(buf.desc, buf.ws) == BLR_OK
    blr_selftest_wait_timeout(buf.desc, buf.ws, 20_000_000)  # 20 ms on a flag nothing sets
    assert blr_workspace_status(buf.desc, buf.ws) == BLR_ERR_TIMEOUT
    buf.fwd()  # the context is still usable and the next forward clears the word
    buf.bwd()
    assert blr_workspace_status(buf.desc, buf.ws) == BLR_OK
    compare(inp, gpu_outputs(buf), oracle_outputs(inp))


def test_autograd_wrapper():
    from paper_2406_12580_gb300 import BDLRUScan
    cfg = I.ScanConfig("autograd", B=3, L=90, D=32, io=I.F32, seed=35, random_h0=True,
                       random_dh_last=True)
    inp = I.make_scan_inputs(cfg)
    dev = "cuda"
    x = torch.tensor(inp.x, device=dev, requires_grad=True)
    gl = torch.tensor(inp.gl, device=dev, requires_grad=True)
    lam = torch.tensor(inp.lam, device=dev, requires_grad=True)
    h0 = torch.tensor(inp.h0, device=dev, requires_grad=True)
    h, h_last = BDLRUScan.apply(x, gl, lam, h0, 1.0)
    loss = (h * torch.tensor(inp.dh, device=dev)).sum() + (h_last * torch.tensor(inp.dh_last, device=dev)).sum()
    loss.backward()
    want = oracle_outputs(inp)
    assert normwise(h.detach().cpu().numpy(), want["h"]) <= 1e-5
    assert normwise(x.grad.cpu().numpy(), want["dx"]) <= 1e-5
    assert normwise(gl.grad.cpu().numpy(), want["dgl"]) <= 1e-5
    assert normwise(lam.grad.cpu().numpy(), want["dlam"]) <= 1e-5
    assert normwise(h0.grad.cpu().numpy(), want["dh0"]) <= 1e-5


def test_binding_rejects_host_tensors():
    from paper_2406_12580_gb300 import Desc, blr_scan_fwd
    x = torch.zeros(1, 4, 8)
    with pytest.raises(ValueError):
        blr_scan_fwd(Desc(1, 4, 8), x, x, x, None, x, None, x)


# The gated layer's merge y = h SiLU(z) (Alg. 1): fused into the serial kernels
# (many chains) and composed with the tiled kernels (few chains), both dtypes.
GATED = [
    dict(B=1, L=1, D=8),
    dict(B=3, L=65, D=72, random_h0=True, random_dh_last=True),
    dict(B=2, L=300, D=16, c=2.0, decay=(0.05, 0.95)),
    dict(B=300, L=203, D=24, random_h0=True, random_dh_last=True),
    dict(B=700, L=37, D=40, decay=(0.05, 0.95), c=0.5),
    dict(B=260, L=1100, D=8, decay=(0.99, 0.9999), random_h0=True),
]


@pytest.mark.parametrize("io", [I.F32, I.BF16])
@pytest.mark.parametrize("case", range(len(GATED)))
def test_gated_small_shapes(io, case):
    inp = I.make_scan_inputs(_cfg(io, 300 + case, gated=True, **GATED[case]))
    buf = gpu_scan_gated(inp)
    compare(inp, gpu_outputs(buf), oracle_outputs(inp))


@pytest.mark.parametrize("k", [1, 2])
def test_gated_config_full_oracle(k):
    """The headline and train-shaped workloads gated, at full size."""
    inp = I.make_scan_inputs(I.scaled(I.CONFIGS[k], gated=True))
    buf = gpu_scan_gated(inp)
    errs = compare(inp, gpu_outputs(buf), oracle_outputs(inp, threads=0))
    print(f"gated config {k}: {errs}")


def test_gated_long_sequence_sampled():
    """The long-sequence workload gated (tiled kernels and the merge kernels),
    on sampled channels."""
    cfg = I.scaled(I.CONFIGS[4], gated=True)
    inp = I.make_scan_inputs(cfg)
    buf = gpu_scan_gated(inp)
    dsel = _sampled_channels(cfg.D)
    errs = compare(inp, gpu_outputs(buf, dsel), oracle_outputs(inp, dsel, threads=0))
    print(f"gated config 4: {errs}")


@pytest.mark.parametrize("io", [I.F32, I.BF16])
def test_gate_math_against_cuda(io):
    """The device gate arithmetic against CUDA's own functions. The step kernel
    evaluates the gates with the same primitives as the scans (sigmoid from
    ex2.approx and rcp.approx in float32, from tanh.approx in the bfloat16
    path; e^l - 1 by its Taylor series where |l| < 0.25, ex2 - 1 beyond;
    sqrt.approx): with h_prev = 1 and x = 0 a step returns alpha, with h_prev = 0
    and x = 1 it returns sqrt(1 - alpha^2) i. Both are compared with the same
    quantities from torch's CUDA float32 operators (expm1f, sigmoid, sqrtf) and
    with float64, over logits in [-30, 30] plus saturating ones, decays
    exp(-softplus(Lambda)) in [0.05, 0.9999] and c in {0.5, 1, 3, 8}.
    Bounds: float32, |d alpha| <= 1e-6 and |d(beta i)| <= (4e-6 + 1e-7 (|rho| +
    |iota|)) |beta i| + 1e-12 (a few units of 2^-23 through each step, and the
    rounding of the sigmoids' exponents); bfloat16, from tanh.approx's
    relative error 2^-11, r and i are off by at most 2^-12, so
    |d alpha| <= |k| 2^-12 + 5e-5 (k = -c softplus(Lambda); 5e-5 covers the
    degree-4 series) and |d(beta i)| <= sqrt(2 |d alpha|) + 2^-12."""
    from paper_2406_12580_gb300 import blr_step, _dtype_code
    B, D = 2048, 64
    g = torch.Generator().manual_seed(11)
    rho = torch.linspace(-30.0, 30.0, B, dtype=torch.float64)
    rho[:8] = torch.tensor([-1e4, -200.0, -80.0, -40.0, 40.0, 80.0, 200.0, 1e4], dtype=torch.float64)
    iota = rho[torch.randperm(B, generator=g)]
    u = torch.linspace(0.05, 0.9999, D, dtype=torch.float64)
    lam = torch.log((1.0 - u) / u).float()
    tdt = torch.float32 if io == I.F32 else torch.bfloat16
    gl = torch.cat([rho[:, None].expand(B, D), iota[:, None].expand(B, D)], dim=1).to(tdt)
    rr, ii = gl[:, :D].double().cpu(), gl[:, D:].double().cpu()  # the rounded logits both sides see
    dev = "cuda"
    gl_d, lam_d = gl.to(dev).contiguous(), lam.to(dev)
    ones = torch.ones(B, D, device=dev)
    zeros = torch.zeros(B, D, device=dev)
    x0, x1 = torch.zeros(B, D, dtype=tdt, device=dev), torch.ones(B, D, dtype=tdt, device=dev)
    for c in (0.5, 1.0, 3.0, 8.0):
        alpha, bi = torch.empty(B, D, device=dev), torch.empty(B, D, device=dev)
        blr_step(B, D, _dtype_code(gl_d), c, ones, x0, gl_d, lam_d, alpha)
        blr_step(B, D, _dtype_code(gl_d), c, zeros, x1, gl_d, lam_d, bi)
        torch.cuda.synchronize()
        alpha, bi = alpha.double().cpu(), bi.double().cpu()
        assert torch.isfinite(alpha).all() and torch.isfinite(bi).all(), c
        k64 = -c * torch.nn.functional.softplus(lam.double())[None, :]
        l64 = k64 * torch.sigmoid(rr)
        a64 = torch.exp(l64)
        bi64 = torch.sqrt(-torch.expm1(2.0 * l64)) * torch.sigmoid(ii)
        # CUDA's float32 functions on the same logits
        r32 = torch.sigmoid(rr.float().to(dev))
        l32 = (-c * torch.nn.functional.softplus(lam_d))[None, :] * r32
        e32 = torch.expm1(l32)
        a32 = (1.0 + e32).double().cpu()
        bi32 = (torch.sqrt(-e32 * (2.0 + e32)) * torch.sigmoid(ii.float().to(dev))).double().cpu()
        da, dbi = (alpha - a64).abs(), (bi - bi64).abs()
        if io == I.F32:
            bound_a = torch.full_like(da, 1e-6)
            # the exponent z log2(e) of the sigmoids is rounded too: 2^-24 |z|
            # relative in each sigmoid, which grows with the logit
            bound_bi = (4e-6 + 1e-7 * (rr.abs() + ii.abs())) * bi64.abs() + 1e-12
        else:
            bound_a = k64.abs().expand(B, D) * 2.0 ** -12 + 5e-5
            bound_bi = torch.sqrt(2.0 * bound_a) + 2.0 ** -12
        worst_a = float((da / bound_a).max())
        worst_bi = float((dbi / bound_bi).max())
        print(f"{io} c={c}: |d alpha| max {float(da.max()):.2e} (CUDA f32 {float((a32 - a64).abs().max()):.2e}), "
              f"|d(beta i)| max {float(dbi.max()):.2e} (CUDA f32 {float((bi32 - bi64).abs().max()):.2e}); "
              f"worst error / bound {worst_a:.3f}, {worst_bi:.3f}")
        assert worst_a <= 1.0 and worst_bi <= 1.0, (io, c, worst_a, worst_bi)


# K recurrent steps per row (blr_steps): io and state dtypes crossed, with and
# without the per-step states, the last state written over the first.
STEPS = [dict(B=1, L=1, D=8), dict(B=3, L=5, D=72), dict(B=1000, L=16, D=64, c=2.0),
         dict(B=65536, L=8, D=64, decay=(0.99, 0.9999))]


def _bf16_round(a):
    return I.bf16_bits_to_f32(I.round_to_bf16(a)).reshape(a.shape)


@pytest.mark.parametrize("state", [I.F32, I.BF16])
@pytest.mark.parametrize("io", [I.F32, I.BF16])
@pytest.mark.parametrize("case", range(len(STEPS)))
def test_steps(case, io, state):
    import oracle
    from paper_2406_12580_gb300 import blr_steps
    from paper_2406_12580_gb300.device import io_code, to_device, torch_io_dtype
    cfg = _cfg(io, 500 + case, random_h0=True, fwd_only=True, **STEPS[case])
    inp = I.make_scan_inputs(cfg)
    B, K, D = cfg.B, cfg.L, cfg.D
    h_prev = inp.h0 if state == I.F32 else _bf16_round(inp.h0)
    x, gl = to_device(inp.io_array("x"), io, "cuda"), to_device(inp.io_array("gl"), io, "cuda")
    lam = to_device(inp.lam, I.F32, "cuda")
    h = torch.from_numpy(h_prev.astype(np.float32)).cuda().to(torch_io_dtype(state))
    h_seq = torch.empty(B, K, D, dtype=torch_io_dtype(io), device="cuda")
    blr_steps(B, K, D, io_code(io), io_code(state), cfg.c, h, x, gl, lam, h, h_seq)  # in place
    torch.cuda.synchronize()
    want_seq, want_out = oracle.load().steps(h_prev, inp.x, inp.gl, inp.lam, c=cfg.c)
    assert normwise(h_seq.float().cpu().numpy(), want_seq) <= TOL[io]
    tol_out = TOL[I.F32] if (io == I.F32 and state == I.F32) else TOL[I.BF16]
    assert normwise(h.float().cpu().numpy(), want_out) <= tol_out
    # without the per-step states, into a separate output; K = 0 copies the state
    h2 = torch.from_numpy(h_prev.astype(np.float32)).cuda().to(torch_io_dtype(state))
    out = torch.empty_like(h2)
    blr_steps(B, K, D, io_code(io), io_code(state), cfg.c, h2, x, gl, lam, out, None)
    blr_steps(B, 0, D, io_code(io), io_code(state), cfg.c, out, None, None, lam, h2, None)
    torch.cuda.synchronize()
    assert torch.equal(out, h)
    assert torch.equal(h2, out)


# Few chains and long bfloat16 sequences: the segmented serial kernels (time
# segments whose maps compose the carries). A partial channel group and a
# ragged last segment, h0 and dh_last entering through the maps, slow decays
# and c != 1, fast decays (the e^l - 1 branch), the shortest sequence that
# segments (at 8 Mi elements), several channel groups per row, and a chain of
# over 300 segments.
SEGMENTED = [
    dict(B=1, L=16500, D=72, random_h0=True, random_dh_last=True),
    dict(B=2, L=20000, D=64, decay=(0.99, 0.9999), c=2.0, random_dh_last=True),
    dict(B=1, L=16384, D=256, decay=(0.05, 0.95), random_h0=True, random_dh_last=True),
    dict(B=64, L=2048, D=64, random_h0=True),
    dict(B=8, L=8200, D=128, random_dh_last=True),
    dict(B=1, L=40000, D=8, decay=(0.99, 0.9999), random_h0=True, random_dh_last=True),
]


def _family(cfg, lengths=False):
    from paper_2406_12580_gb300 import Desc, blr_scan_family
    return blr_scan_family(Desc(cfg.B, cfg.L, cfg.D, 0 if cfg.io == I.F32 else 1, cfg.c), lengths)


@pytest.mark.parametrize("case", range(len(SEGMENTED)))
def test_segmented(case):
    from paper_2406_12580_gb300 import FAMILY_SEGMENTED
    inp = I.make_scan_inputs(_cfg(I.BF16, 500 + case, **SEGMENTED[case]))
    assert _family(inp.cfg) == FAMILY_SEGMENTED
    compare(inp, gpu_outputs(gpu_scan(inp)), oracle_outputs(inp))


@pytest.mark.parametrize("case", [0, 2, 3])
def test_segmented_gated(case):
    inp = I.make_scan_inputs(_cfg(I.BF16, 520 + case, gated=True, **SEGMENTED[case]))
    compare(inp, gpu_outputs(gpu_scan_gated(inp)), oracle_outputs(inp))


def test_segmented_workspace_tags():
    """A segmented backward refuses a workspace that a tiled forward of the
    same shape filled (the _varlen forms run tiled here), and the tiled
    backward refuses a segmented forward's."""
    from paper_2406_12580_gb300 import (BLR_ERR_WORKSPACE, BLR_OK, FAMILY_TILED,
                                        blr_workspace_status)
    from paper_2406_12580_gb300.device import ScanBuffers
    cfg = _cfg(I.BF16, 530, **SEGMENTED[0])
    assert _family(cfg, lengths=True) == FAMILY_TILED
    inp = I.make_scan_inputs(cfg)
    buf = ScanBuffers.from_inputs(inp)
    full = torch.full((cfg.B,), cfg.L, dtype=torch.int32, device="cuda")
    buf.fwd_varlen(full)  # tiled kernels, all rows full length
    buf.dx.fill_(3.0)
    buf.bwd()
    assert blr_workspace_status(buf.desc, buf.ws) == BLR_ERR_WORKSPACE
    assert torch.all(buf.dx == 3.0)
    buf.fwd()
    buf.bwd()
    assert blr_workspace_status(buf.desc, buf.ws) == BLR_OK
    compare(inp, gpu_outputs(buf), oracle_outputs(inp))
    buf.bwd_varlen(full)  # tiled backward after a segmented forward: refused
    assert blr_workspace_status(buf.desc, buf.ws) == BLR_ERR_WORKSPACE


@pytest.mark.parametrize("io,shape", [(I.F32, dict(B=300, L=130, D=40)),
                                      (I.F32, dict(B=3, L=300, D=72)),
                                      (I.BF16, dict(B=1, L=16500, D=72))])
def test_backward_without_workspace(io, shape):
    """ws = NULL: the backward recomputes the forward's carries in the library's
    scratch and gives the results of a backward from the forward's workspace,
    plain, gated and with row lengths, on the three kernel families."""
    from paper_2406_12580_gb300 import (BLR_OK, blr_scan_bwd, blr_scan_bwd_gated,
                                        blr_scan_bwd_varlen, blr_workspace_status)
    from paper_2406_12580_gb300.device import ScanBuffers
    cfg = _cfg(io, 950, random_h0=True, random_dh_last=True, **shape)
    inp = I.make_scan_inputs(cfg)
    buf = ScanBuffers.from_inputs(inp)
    lengths = torch.from_numpy(np.random.default_rng(3).integers(0, cfg.L + 1, size=cfg.B)
                               .astype(np.int32)).cuda()
    outs = lambda: [t.clone() for t in (buf.dx, buf.dgl, buf.dlam, buf.dh0)]  # noqa: E731
    z = torch.randn_like(buf.x)
    dz = torch.zeros_like(buf.x)
    for mode in ("plain", "gated", "varlen"):
        for t in (buf.dx, buf.dgl, dz):
            t.zero_()
        if mode == "plain":
            buf.fwd()
            buf.bwd()
        elif mode == "gated":
            buf.fwd()  # a plain forward's workspace serves the gated backward
            blr_scan_bwd_gated(buf.desc, buf.dh, buf.dh_last, buf.x, buf.gl, buf.lam, buf.h0, z,
                               buf.dx, buf.dgl, dz, buf.dlam, buf.dh0, buf.ws)
        else:
            buf.fwd_varlen(lengths)
            buf.bwd_varlen(lengths)
        torch.cuda.synchronize()
        want = outs() + ([dz.clone()] if mode == "gated" else [])
        for t in (buf.dx, buf.dgl, buf.dlam, buf.dh0, dz):
            t.fill_(7.0)
        buf.ws.zero_()  # nothing of the forward is left for the backward
        if mode == "plain":
            blr_scan_bwd(buf.desc, buf.dh, buf.dh_last, buf.x, buf.gl, buf.lam, buf.h0, buf.dx,
                         buf.dgl, buf.dlam, buf.dh0, None)
        elif mode == "gated":
            blr_scan_bwd_gated(buf.desc, buf.dh, buf.dh_last, buf.x, buf.gl, buf.lam, buf.h0, z,
                               buf.dx, buf.dgl, dz, buf.dlam, buf.dh0, None)
        else:
            for t in (buf.dx, buf.dgl):
                t.copy_(want[0] if t is buf.dx else want[1])  # the padding is never written
            blr_scan_bwd_varlen(buf.desc, lengths, buf.dh, buf.dh_last, buf.x, buf.gl, buf.lam,
                                buf.h0, buf.dx, buf.dgl, buf.dlam, buf.dh0, None)
        torch.cuda.synchronize()
        assert blr_workspace_status(buf.desc, None) == BLR_OK
        got = outs() + ([dz.clone()] if mode == "gated" else [])
        for g, w in zip(got, want):
            # the same kernels: float32 results agree up to the order of float
            # atomics and of the tiled look-back's combines, which can move a
            # bfloat16 output by one unit in its last place
            tol = 2.0 ** -7 if g.dtype == torch.bfloat16 else 1e-6
            assert normwise(g.float().cpu().numpy(), w.float().cpu().numpy()) <= tol, mode


# Rows of their own lengths (blr_scan_*_varlen): sequences right-aligned in
# their rows (left padding), padding never read or written; both kernel
# families, empty and full rows included.
VARLEN = [dict(B=3, L=65, D=72, random_h0=True, random_dh_last=True),
          dict(B=2, L=300, D=16),
          dict(B=300, L=203, D=24, random_h0=True, random_dh_last=True),
          dict(B=700, L=37, D=40, decay=(0.05, 0.95), c=2.0),
          dict(B=260, L=1100, D=8, decay=(0.99, 0.9999), random_h0=True)]


@pytest.mark.parametrize("io", [I.F32, I.BF16])
@pytest.mark.parametrize("case", range(len(VARLEN)))
def test_varlen(io, case):
    import oracle
    from paper_2406_12580_gb300.device import ScanBuffers
    cfg = _cfg(io, 600 + case, **VARLEN[case])
    inp = I.make_scan_inputs(cfg)
    B, L, D = cfg.B, cfg.L, cfg.D
    lengths = np.random.default_rng(case).integers(0, L + 1, size=B).astype(np.int32)
    lengths[0] = L
    lengths[1] = 0
    lengths[-1] = min(L, 3)
    buf = ScanBuffers.from_inputs(inp)
    for t in (buf.h, buf.dx, buf.dgl):
        t.fill_(float("nan"))
    lt = torch.from_numpy(lengths).cuda()
    buf.fwd_varlen(lt)
    buf.bwd_varlen(lt)
    torch.cuda.synchronize()
    orc = oracle.load()
    h, h_last = orc.fwd_varlen(lengths, inp.x, inp.gl, inp.lam, inp.h0, c=cfg.c)
    dx, dgl, dlam, dh0 = orc.bwd_varlen(lengths, inp.dh, inp.x, inp.gl, inp.lam, inp.h0,
                                        inp.dh_last, c=cfg.c)
    got = gpu_outputs(buf)
    real = ~np.isnan(h)
    real2 = np.concatenate([real, real], axis=2)
    tol = TOL[io]
    # the padding keeps what the caller left there: nothing was written
    assert np.isnan(got["h"][~real]).all() and np.isnan(got["dx"][~real]).all()
    assert np.isnan(got["dgl"][~real2]).all()
    assert normwise(got["h"][real], h[real]) <= tol
    assert normwise(got["dx"][real], dx[real]) <= tol
    assert normwise(got["dgl"][real2], dgl[real2]) <= tol
    for k, w in (("h_last", h_last), ("dlam", dlam), ("dh0", dh0)):
        assert normwise(got[k], w) <= tol, k


# Seeded random problems across the whole surface: dtype, shape, h0 / dh_last,
# c, decays, row lengths and the gated merge drawn at random (fixed seeds).
def _fuzz_case(seed):
    rng = np.random.default_rng(seed)
    io = [I.F32, I.BF16][rng.integers(2)]
    B = int(rng.choice([1, 2, 5, 40, 300, 700]))
    D = int(8 * rng.integers(1, 17))
    L = int(rng.integers(1, max(2, min(400, 1_000_000 // (B * D)))))  # the oracle stays quick
    lo = float(rng.choice([0.05, 0.5, 0.9, 0.99]))
    kw = dict(B=B, L=L, D=D, decay=(lo, min(0.9999, lo + 0.09)), c=float(rng.choice([0.5, 1.0, 3.0])),
              random_h0=bool(rng.integers(2)), random_dh_last=bool(rng.integers(2)),
              gate_std=float(rng.choice([0.5, 1.0, 3.0])))
    mode = ["plain", "gated", "varlen"][rng.integers(3)]
    return io, kw, mode, rng


@pytest.mark.parametrize("seed", range(24))
def test_fuzz(seed):
    import oracle
    io, kw, mode, rng = _fuzz_case(seed)
    cfg = _cfg(io, 700 + seed, gated=(mode == "gated"), **kw)
    inp = I.make_scan_inputs(cfg)
    if mode == "gated":
        compare(inp, gpu_outputs(gpu_scan_gated(inp)), oracle_outputs(inp))
    elif mode == "plain":
        compare(inp, gpu_outputs(gpu_scan(inp)), oracle_outputs(inp))
    else:
        from paper_2406_12580_gb300.device import ScanBuffers
        lengths = rng.integers(0, cfg.L + 1, size=cfg.B).astype(np.int32)
        buf = ScanBuffers.from_inputs(inp)
        for t in (buf.h, buf.dx, buf.dgl):
            t.zero_()  # the padding is not written: keep it defined
        lt = torch.from_numpy(lengths).cuda()
        buf.fwd_varlen(lt)
        buf.bwd_varlen(lt)
        torch.cuda.synchronize()
        orc = oracle.load()
        h, h_last = orc.fwd_varlen(lengths, inp.x, inp.gl, inp.lam, inp.h0, c=cfg.c)
        dx, dgl, dlam, dh0 = orc.bwd_varlen(lengths, inp.dh, inp.x, inp.gl, inp.lam, inp.h0,
                                            inp.dh_last, c=cfg.c)
        got = gpu_outputs(buf)
        real = ~np.isnan(h)
        real2 = np.concatenate([real, real], axis=2)
        tol = TOL[io]
        assert normwise(got["h"][real], h[real]) <= tol
        assert normwise(got["dx"][real], dx[real]) <= tol
        assert normwise(got["dgl"][real2], dgl[real2]) <= tol
        for k, w in (("h_last", h_last), ("dlam", dlam), ("dh0", dh0)):
            assert normwise(got[k], w) <= tol, k


@pytest.mark.parametrize("io,shape", [(I.F32, dict(B=300, L=130, D=40)),
                                      (I.F32, dict(B=3, L=300, D=72)),
                                      (I.BF16, dict(B=1, L=16500, D=72))])
def test_graph_capture_replays_eager(io, shape):
    """The forward and backward captured into a CUDA graph (no host work is
    needed between them) replay to the eager results, on the three kernel
    families."""
    inp = I.make_scan_inputs(_cfg(io, 900, random_h0=True, random_dh_last=True, **shape))
    eager = gpu_outputs(gpu_scan(inp))
    from paper_2406_12580_gb300.device import ScanBuffers
    buf = ScanBuffers.from_inputs(inp)
    buf.fwd()
    buf.bwd()  # first calls outside capture (per-device setup)
    torch.cuda.synchronize()
    for t in (buf.h, buf.dx, buf.dgl, buf.dlam):
        t.zero_()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(g, stream=side):
            buf.fwd()
            buf.bwd()
    torch.cuda.current_stream().wait_stream(side)
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    got = gpu_outputs(buf)
    # the same kernels, so the same values up to the order of float atomics
    # (dLambda) and of look-back combines: a look-back folds whichever
    # predecessors have published when it reads, so float32 carries may differ
    # in their last bits between calls, and a bfloat16 output by one unit in
    # its last place (at most 2^-7 of its magnitude) where such a carry sits at
    # a rounding boundary
    tol = 1e-6 if io == I.F32 else 2.0 ** -7
    for k in eager:
        assert normwise(got[k], eager[k]) <= tol, k
