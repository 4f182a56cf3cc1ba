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
import pytest

from gpu_common import normwise
from paper_2406_12580_gb300 import inputs as I

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, but never run there
    pytest.skip("no CUDA device", allow_module_level=True)


def _both(cfg):
    """blr_scan_fwd_noalloc against blr_scan_fwd with a caller workspace on the
    same inputs, and both against the oracle. The serial kernels are
    deterministic: there the outputs must be bit for bit the same. The kernels
    that chain tiles with a look-back fold whichever predecessors have
    published when they read, so their float32 states may differ in the last
    bits between calls, and a bfloat16 output by one unit in its last place
    (at most 2^-7 of its magnitude)."""
    from paper_2406_12580_gb300 import FAMILY_SERIAL, blr_scan_family, blr_scan_fwd_noalloc
    from paper_2406_12580_gb300.device import ScanBuffers
    inp = I.make_scan_inputs(cfg)
    buf = ScanBuffers.from_inputs(inp, with_bwd=False)
    buf.fwd()  # the ordinary entry point, caller workspace
    h = torch.full_like(buf.h, float("nan"))
    h_last = torch.full_like(buf.h_last, float("nan"))
    blr_scan_fwd_noalloc(buf.desc, buf.x, buf.gl, buf.lam, buf.h0, h, h_last)
    torch.cuda.synchronize()
    assert torch.isfinite(h.float()).all() and torch.isfinite(h_last).all()
    if blr_scan_family(buf.desc) == FAMILY_SERIAL:
        assert torch.equal(h, buf.h) and torch.equal(h_last, buf.h_last)
    else:
        step = 1e-6 if cfg.io == I.F32 else 2.0 ** -7
        assert normwise(h.float().cpu().numpy(), buf.h.float().cpu().numpy()) <= step
        assert normwise(h_last.cpu().numpy(), buf.h_last.cpu().numpy()) <= 1e-6
    return inp, h, h_last


def _against_oracle(inp, h, h_last):
    from gpu_common import compare, oracle_outputs
    want = oracle_outputs(inp)
    compare(inp, {"h": h.double().cpu().numpy(), "h_last": h_last.double().cpu().numpy()},
            {"h": want["h"], "h_last": want["h_last"]})


def test_noalloc_forward_matches_workspace_forward_on_consecutive_calls():
    # different problems in a row, then the first again: each call must start
    # from a cleared scratch, whatever the previous call left in it
    a = I.ScanConfig("noalloc a", B=3, L=700, D=64, io=I.F32, seed=41, random_h0=True)
    b = I.ScanConfig("noalloc b", B=4, L=300, D=72, io=I.BF16, seed=42)
    c = I.ScanConfig("noalloc c", B=300, L=50, D=64, io=I.BF16, seed=44, random_h0=True)
    _against_oracle(*_both(a))
    _against_oracle(*_both(b))
    _against_oracle(*_both(c))
    _both(a)
    _both(c)


def test_noalloc_forward_at_a_long_sequence_size():
    # the long-sequence workload, 8 x 32768 x 512 bfloat16 (its workspace,
    # about 113 MiB, fits the 128 MiB scratch)
    cfg = I.ScanConfig("noalloc long", B=8, L=32768, D=512, io=I.BF16, seed=43, decay=(0.99, 0.9999))
    _both(cfg)
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
