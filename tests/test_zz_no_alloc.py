"""GPU: the forward scan that allocates nothing, blr_scan_fwd_noalloc.

Some callers cannot allocate the workspace blr_scan_fwd needs: code running
inside CUDA stream capture, plugins whose host framework owns every device
allocation, serving loops that forbid allocator calls. blr_scan_fwd_noalloc
runs the same forward scan on a scratch array the library keeps in device
memory. These tests call it through the C ABI and check that it returns what
blr_scan_fwd returns with a caller workspace, on consecutive calls (the calls
share the one scratch array, so the second must not see the first's state).

The file is named to be collected last, so that a run stopping at the first
failure has run every other test before it.
"""
import numpy as np
import pytest

from gpu_common import TOL, normwise
from paper_2406_12580_gb300 import inputs as I

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, but never run there
    pytest.skip("no CUDA device", allow_module_level=True)


def _both(cfg):
    from paper_2406_12580_gb300 import blr_scan_fwd_noalloc
    from paper_2406_12580_gb300.device import ScanBuffers
    inp = I.make_scan_inputs(cfg)
    buf = ScanBuffers.from_inputs(inp, with_bwd=False)
    buf.fwd()  # the ordinary entry point, caller workspace
    h = torch.full_like(buf.h, float("nan"))
    h_last = torch.full_like(buf.h_last, float("nan"))
    blr_scan_fwd_noalloc(buf.desc, buf.x, buf.gl, buf.lam, buf.h0, h, h_last)
    torch.cuda.synchronize()
    tol = TOL[cfg.io]
    got_h, want_h = h.float().cpu().numpy(), buf.h.float().cpu().numpy()
    assert np.isfinite(got_h).all()
    assert normwise(got_h, want_h) <= tol
    assert normwise(h_last.cpu().numpy(), buf.h_last.cpu().numpy()) <= tol


def test_noalloc_forward_matches_workspace_forward_on_consecutive_calls():
    # two different problems, then the first again: each call must start from
    # a cleared scratch, whatever the previous call left in it
    a = I.ScanConfig("noalloc a", B=3, L=700, D=64, io=I.F32, seed=41, random_h0=True)
    b = I.ScanConfig("noalloc b", B=4, L=300, D=72, io=I.BF16, seed=42)
    _both(a)
    _both(b)
    _both(a)


def test_noalloc_forward_at_a_long_sequence_size():
    # the long-sequence workload, 8 x 32768 x 512 bfloat16 (segmented kernels;
    # its workspace, about 94 MB, fits the 128 MiB scratch)
    cfg = I.ScanConfig("noalloc long", B=8, L=32768, D=512, io=I.BF16, seed=43, decay=(0.99, 0.9999))
    _both(cfg)


def test_noalloc_rejects_problems_above_its_scratch():
    from paper_2406_12580_gb300 import BLR_ERR_UNSUPPORTED, Desc, _lib
    import ctypes
    lib = _lib.load()
    desc = Desc(64, 100000, 512)  # needs far more than 128 MiB of scratch
    assert lib.blr_workspace_bytes(ctypes.byref(desc)) > (128 << 20)
    st = lib.blr_scan_fwd_noalloc(ctypes.byref(desc), None, None, None, None, None, None, None)
    assert st == BLR_ERR_UNSUPPORTED
    assert b"static scratch" in lib.blr_last_error_string()
