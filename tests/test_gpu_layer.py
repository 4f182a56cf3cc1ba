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
