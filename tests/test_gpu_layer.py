"""GPU: the gated recurrent layer of Alg. 1 (``paper_2406_12580_gb300.layer``) on
the library's fused scan-and-merge kernels, against the same layer written with
plain torch operations in float64 on the CPU (the scan as a step-by-step loop),
outputs and every gradient."""
import copy

import numpy as np
import pytest

from gpu_common import normwise

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, but never run there
    pytest.skip("no CUDA device", allow_module_level=True)


def reference_forward(layer, h):
    """Alg. 1 with torch operators only; the BD-LRU as the Sec. 3.2 recurrence."""
    B, L, _ = h.shape
    hx, hz = layer.in_proj(h).split(layer.ed, dim=-1)
    xc = layer.conv(hx.transpose(1, 2))[..., :L].transpose(1, 2)
    x = torch.nn.functional.silu(xc)
    rho, iota = layer.gate_proj(x).split(layer.ed, dim=-1)
    r, i = torch.sigmoid(rho), torch.sigmoid(iota)
    alpha = torch.exp(-layer.c * torch.nn.functional.softplus(layer.lam) * r)
    beta = torch.sqrt(1.0 - alpha * alpha) * i
    state = torch.zeros(B, layer.ed, dtype=x.dtype)
    hs = []
    for t in range(L):
        state = alpha[:, t] * state + beta[:, t] * x[:, t]
        hs.append(state)
    y = torch.stack(hs, dim=1) * torch.nn.functional.silu(hz)
    return layer.out_proj(y)


@pytest.mark.parametrize("shape", [(3, 40, 16, 2), (260, 33, 16, 2), (2, 300, 8, 1)])
def test_layer_matches_torch_reference(shape):
    from paper_2406_12580_gb300.layer import GatedRecurrentLayer
    torch.backends.cudnn.allow_tf32 = False
    torch.backends.cuda.matmul.allow_tf32 = False
    B, L, D, E = shape
    torch.manual_seed(7)
    layer = GatedRecurrentLayer(D, expand=E, c=1.0, device="cuda")
    ref = copy.deepcopy(layer).double().cpu()
    h = torch.randn(B, L, D, device="cuda", requires_grad=True)
    g = torch.randn(B, L, D, device="cuda")
    out = layer(h)
    (out * g).sum().backward()
    h64 = h.detach().double().cpu().requires_grad_(True)
    out64 = reference_forward(ref, h64)
    (out64 * g.double().cpu()).sum().backward()
    assert normwise(out.detach().cpu().numpy(), out64.detach().numpy()) <= 1e-5
    assert normwise(h.grad.cpu().numpy(), h64.grad.numpy()) <= 1e-5
    for (name, p), (_, q) in zip(layer.named_parameters(), ref.named_parameters()):
        assert normwise(p.grad.cpu().numpy(), q.grad.numpy()) <= 1e-5, name


def test_layer_bf16_close_to_f32():
    from paper_2406_12580_gb300.layer import GatedRecurrentLayer
    torch.manual_seed(8)
    layer = GatedRecurrentLayer(32, expand=2, device="cuda")
    h = torch.randn(256, 50, 32, device="cuda")
    want = layer(h).detach()
    got = copy.deepcopy(layer).to(torch.bfloat16)(h.to(torch.bfloat16)).float().detach()
    assert np.isfinite(got.cpu().numpy()).all()
    assert normwise(got.cpu().numpy(), want.cpu().numpy()) <= 5e-2


@pytest.mark.parametrize("io,B,L,D", [("f32", 300, 40, 64), ("f32", 3, 150, 72),
                                     ("bf16", 300, 40, 64), ("bf16", 3, 150, 72)])
def test_gated_scan_autograd_against_oracle(io, B, L, D):
    """BDLRUGatedScan (the autograd function the layer runs: the BD-LRU and the
    merge with SiLU(z) of Alg. 1, fused) against the oracle's gated forward and
    backward: y, h_last and the gradients of x, the gate logits, Lambda, z and h0."""
    from gpu_common import compare
    import oracle
    from paper_2406_12580_gb300 import inputs as I
    from paper_2406_12580_gb300.device import to_device
    from paper_2406_12580_gb300.layer import BDLRUGatedScan
    cfg = I.ScanConfig(f"gated autograd {io} B={B} L={L} D={D}", B, L, D, io, seed=77,
                       random_h0=True, random_dh_last=True, gated=True)
    inp = I.make_scan_inputs(cfg)
    dev = torch.device("cuda")
    leaf = lambda name: to_device(inp.io_array(name), io, dev).requires_grad_(True)  # noqa: E731
    x, gl, z = leaf("x"), leaf("gl"), leaf("z")
    lam = to_device(inp.lam, "f32", dev).requires_grad_(True)
    h0 = to_device(inp.h0, "f32", dev).requires_grad_(True)
    y, h_last = BDLRUGatedScan.apply(x, gl, lam, z, h0, 1.0)
    dy = to_device(inp.io_array("dh"), io, dev)
    dh_last = to_device(inp.dh_last, "f32", dev)
    torch.autograd.backward([y, h_last], [dy, dh_last])
    orc = oracle.load()
    want_y, want_hl = orc.fwd_gated(inp.x, inp.gl, inp.lam, inp.z, inp.h0)
    dx, dgl, dlam, dh0, dz = orc.bwd_gated(inp.dh, inp.x, inp.gl, inp.lam, inp.z, inp.h0, inp.dh_last)
    f64 = lambda t: t.detach().double().cpu().numpy()  # noqa: E731
    got = {"h": f64(y), "h_last": f64(h_last), "dx": f64(x.grad), "dgl": f64(gl.grad),
           "dlam": f64(lam.grad), "dh0": f64(h0.grad), "dz": f64(z.grad)}
    want = {"h": want_y, "h_last": want_hl, "dx": dx, "dgl": dgl, "dlam": dlam, "dh0": dh0, "dz": dz}
    compare(inp, got, want)


class _Filter:
    """The synthetic sequence task: the target is a causal exponential filter
    of a fixed linear map of the input, y_t = sum_{j<=t} 0.8^(t-j) A h_j / 3,
    which a BD-LRU layer can represent (a decay per channel and a readout)."""

    def __init__(self, d, seed):
        g = torch.Generator().manual_seed(seed)
        self.A = torch.randn(d, d, generator=g, dtype=torch.float64) / d ** 0.5
        self.g = g

    def batch(self, B, L, d):
        h = torch.randn(B, L, d, generator=self.g, dtype=torch.float64)
        u = h @ self.A.T
        y = torch.zeros_like(u)
        acc = torch.zeros(B, d, dtype=torch.float64)
        for t in range(L):
            acc = 0.8 * acc + u[:, t]
            y[:, t] = acc / 3.0
        return h, y


def test_layer_trains_on_a_synthetic_sequence_task():
    """A few hundred Adam steps (lr 1e-3, the paper's optimiser settings) of the
    layer on the filter task: the loss falls to below half its starting value
    (measured: 0.270 -> 0.105 over 300 steps, 2.6x)."""
    from paper_2406_12580_gb300.layer import GatedRecurrentLayer
    torch.manual_seed(11)
    d, B, L = 16, 64, 64
    layer = GatedRecurrentLayer(d, expand=2, device="cuda")
    opt = torch.optim.Adam(layer.parameters(), lr=1e-3)
    task = _Filter(d, 12)
    losses = []
    for _ in range(300):
        h, y = task.batch(B, L, d)
        out = layer(h.float().cuda())
        loss = torch.mean((out - y.float().cuda()) ** 2)
        opt.zero_grad()
        loss.backward()
        opt.step()
        losses.append(float(loss))
    first, last = np.mean(losses[:10]), np.mean(losses[-10:])
    print(f"loss {first:.4f} -> {last:.4f} ({first / last:.1f}x)")
    assert np.isfinite(losses).all()
    assert last <= first / TRAIN_FACTOR, (first, last)


TRAIN_FACTOR = 2.0


def test_first_adam_updates_match_float64_reference():
    """Three Adam steps of the layer on the GPU (float32, the library's kernels)
    against the same steps of a float64 CPU copy (torch operators, the scan as
    the Sec. 3.2 recurrence): every parameter after every step within 1e-5."""
    from paper_2406_12580_gb300.layer import GatedRecurrentLayer
    torch.backends.cudnn.allow_tf32 = False
    torch.backends.cuda.matmul.allow_tf32 = False
    torch.manual_seed(13)
    d, B, L = 16, 4, 20
    layer = GatedRecurrentLayer(d, expand=2, device="cuda")
    ref = copy.deepcopy(layer).double().cpu()
    opt = torch.optim.Adam(layer.parameters(), lr=1e-3)
    opt_ref = torch.optim.Adam(ref.parameters(), lr=1e-3)
    task = _Filter(d, 14)
    for step in range(3):
        h, y = task.batch(B, L, d)
        loss = torch.mean((layer(h.float().cuda()) - y.float().cuda()) ** 2)
        opt.zero_grad()
        loss.backward()
        opt.step()
        loss_ref = torch.mean((reference_forward(ref, h) - y) ** 2)
        opt_ref.zero_grad()
        loss_ref.backward()
        opt_ref.step()
        for (name, p), (_, q) in zip(layer.named_parameters(), ref.named_parameters()):
            err = normwise(p.detach().cpu().numpy(), q.detach().numpy())
            assert err <= 1e-5, (step, name, err)
