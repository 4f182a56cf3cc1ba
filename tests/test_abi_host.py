"""CPU: the C-ABI library loads, exports every entry point include/blr.h declares,
and rejects bad arguments on the host before anything reaches a GPU.

Only validation failures are exercised here: every call below returns before
the library makes any CUDA call, so the fake (never dereferenced) addresses
used as pointers are never handed to a device."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2406_12580_gb300 import _lib
from paper_2406_12580_gb300 import build as blr_build

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "blr.h")

FAKE = 0x7f0000000000  # 256-byte aligned address, never dereferenced


@pytest.fixture(scope="module")
def lib():
    if blr_build.stale():
        blr_build.build()
    return _lib.load()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^BLR_API\s+[\w\s\*]*?\b(blr_\w+)\s*\(", text, re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("blr_scan_fwd", "blr_scan_bwd", "blr_step", "blr_workspace_bytes", "blr_status_string"):
        assert n in names
    assert set(names) == set(_lib.SIGNATURES), "ctypes table out of sync with include/blr.h"


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", _lib.library_path()], check=True,
                         stdout=subprocess.PIPE, text=True).stdout
    exported = set(re.findall(r"\sT\s+(\w+)$", out, re.M))
    for name in declared_functions():
        assert name in exported, name
        assert getattr(lib, name) is not None
    # nothing else leaks out of the library
    assert {e for e in exported if e.startswith("blr_")} == set(declared_functions())


def D(B, L, Dd, io=0, c=1.0):
    return _lib.blr_desc(B, L, Dd, io, c)


def fwd(lib, desc, x=FAKE, gl=FAKE, lam=FAKE, h0=None, h=FAKE, h_last=None, ws=FAKE, ws_bytes=None):
    if ws_bytes is None:
        ws_bytes = lib.blr_workspace_bytes(ctypes.byref(desc)) if desc is not None else 0
    dp = ctypes.byref(desc) if desc is not None else None
    return lib.blr_scan_fwd(dp, x, gl, lam, h0, h, h_last, ws, ws_bytes, None)


def test_fwd_validation(lib):
    assert lib.blr_scan_fwd(None, FAKE, FAKE, FAKE, None, FAKE, None, FAKE, 1 << 20, None) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(-1, 4, 8)) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(1, -4, 8)) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(1, 4, 8, io=7)) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(1, 4, 8, c=0.0)) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(1, 4, 8, c=float("nan"))) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(1, 4, 8, c=float("inf"))) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(1, 4, 12)) == _lib.BLR_ERR_UNSUPPORTED
    assert b"multiple of 8" in lib.blr_last_error_string()
    # empty batch or channels: a no-op that touches nothing, even with NULL pointers
    assert fwd(lib, D(0, 4, 8), x=None, gl=None, lam=None, h=None, ws=None) == _lib.BLR_OK
    assert fwd(lib, D(3, 4, 0), x=None, gl=None, lam=None, h=None, ws=None) == _lib.BLR_OK
    # required pointers and alignment
    assert fwd(lib, D(2, 4, 8), x=None) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), gl=None) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), lam=None) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), ws=None) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), x=FAKE + 4) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), gl=FAKE + 8) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), h=FAKE + 2) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), lam=FAKE + 4) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), h0=FAKE + 2) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), h_last=FAKE + 1) == _lib.BLR_ERR_INVALID_ARG
    assert fwd(lib, D(2, 4, 8), ws=FAKE + 8) == _lib.BLR_ERR_INVALID_ARG
    desc = D(2, 4, 8)
    need = lib.blr_workspace_bytes(ctypes.byref(desc))
    assert fwd(lib, desc, ws_bytes=need - 1) == _lib.BLR_ERR_INVALID_ARG
    assert b"ws_bytes" in lib.blr_last_error_string()


def bwd(lib, desc, **kw):
    args = dict(dh=FAKE, dh_last=None, x=FAKE, gl=FAKE, lam=FAKE, h0=None, dx=FAKE, dgl=FAKE,
                dlam=FAKE, dh0=None, ws=FAKE, ws_bytes=None)
    args.update(kw)
    if args["ws_bytes"] is None:
        args["ws_bytes"] = lib.blr_workspace_bytes(ctypes.byref(desc))
    return lib.blr_scan_bwd(ctypes.byref(desc), args["dh"], args["dh_last"], args["x"], args["gl"],
                            args["lam"], args["h0"], args["dx"], args["dgl"], args["dlam"],
                            args["dh0"], args["ws"], args["ws_bytes"], None)


def test_bwd_validation(lib):
    assert bwd(lib, D(2, 4, 12)) == _lib.BLR_ERR_UNSUPPORTED
    assert bwd(lib, D(2, 4, 8, c=-1.0)) == _lib.BLR_ERR_INVALID_ARG
    for name in ("dh", "x", "gl", "lam", "dx", "dgl", "dlam"):
        assert bwd(lib, D(2, 4, 8), **{name: None}) == _lib.BLR_ERR_INVALID_ARG, name
    # without a workspace the backward recomputes the carries in the library's
    # 128 MiB scratch; a problem that does not fit is refused before anything
    # is enqueued
    big = D(64, 100000, 512)
    assert lib.blr_workspace_bytes(ctypes.byref(big)) > (128 << 20)
    assert bwd(lib, big, ws=None, ws_bytes=0) == _lib.BLR_ERR_UNSUPPORTED
    assert b"static scratch" in lib.blr_last_error_string()
    for name in ("dh", "x", "gl", "dx", "dgl", "lam"):
        assert bwd(lib, D(2, 4, 8), **{name: FAKE + 8}) == _lib.BLR_ERR_INVALID_ARG, name
    for name in ("dh_last", "h0", "dh0", "dlam"):
        assert bwd(lib, D(2, 4, 8), **{name: FAKE + 2}) == _lib.BLR_ERR_INVALID_ARG, name
    assert bwd(lib, D(2, 4, 8), ws_bytes=16) == _lib.BLR_ERR_INVALID_ARG
    assert bwd(lib, D(0, 4, 8), dh=None, x=None, gl=None, lam=None, dx=None, dgl=None, dlam=None,
               ws=None) == _lib.BLR_OK


def fwd_gated(lib, desc, z=FAKE, y=FAKE):
    ws_bytes = lib.blr_workspace_bytes(ctypes.byref(desc))
    return lib.blr_scan_fwd_gated(ctypes.byref(desc), FAKE, FAKE, FAKE, None, z, y, None, FAKE,
                                  ws_bytes, None)


def bwd_gated(lib, desc, z=FAKE, dz=FAKE, dy=FAKE):
    ws_bytes = lib.blr_workspace_bytes(ctypes.byref(desc))
    return lib.blr_scan_bwd_gated(ctypes.byref(desc), dy, None, FAKE, FAKE, FAKE, None, z, FAKE,
                                  FAKE, dz, FAKE, None, FAKE, ws_bytes, None)


def test_gated_validation(lib):
    assert fwd_gated(lib, D(2, 4, 8), z=None) == _lib.BLR_ERR_INVALID_ARG
    assert b"z is NULL" in lib.blr_last_error_string()
    assert fwd_gated(lib, D(2, 4, 8), z=FAKE + 8) == _lib.BLR_ERR_INVALID_ARG
    assert fwd_gated(lib, D(2, 4, 8), y=FAKE + 2) == _lib.BLR_ERR_INVALID_ARG
    assert fwd_gated(lib, D(2, 4, 12), z=None) == _lib.BLR_ERR_UNSUPPORTED  # the shape first
    assert fwd_gated(lib, D(0, 4, 8), z=None, y=None) == _lib.BLR_OK
    assert bwd_gated(lib, D(2, 4, 8), z=None) == _lib.BLR_ERR_INVALID_ARG
    assert bwd_gated(lib, D(2, 4, 8), dz=None) == _lib.BLR_ERR_INVALID_ARG
    assert b"dz is NULL" in lib.blr_last_error_string()
    assert bwd_gated(lib, D(2, 4, 8), dz=FAKE + 4) == _lib.BLR_ERR_INVALID_ARG
    assert bwd_gated(lib, D(2, 4, 8), dy=None) == _lib.BLR_ERR_INVALID_ARG
    assert b"dy is NULL" in lib.blr_last_error_string()


def test_steps_validation(lib):
    f = lambda B, K, Dd, io=0, st=0, c=1.0, hp=FAKE, x=FAKE, gl=FAKE, lam=FAKE, ho=FAKE, hs=None: \
        lib.blr_steps(B, K, Dd, io, st, c, hp, x, gl, lam, ho, hs, None)  # noqa: E731
    assert f(-1, 2, 8) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, -2, 8) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, 2, 8, io=2) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, 2, 8, st=5) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, 2, 8, c=0.0) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, 2, 12) == _lib.BLR_ERR_UNSUPPORTED
    for name in ("hp", "x", "gl", "lam", "ho"):
        assert f(4, 2, 8, **{name: None}) == _lib.BLR_ERR_INVALID_ARG, name
        assert f(4, 2, 8, **{name: FAKE + 8}) == _lib.BLR_ERR_INVALID_ARG, name
    assert f(4, 2, 8, hs=FAKE + 4) == _lib.BLR_ERR_INVALID_ARG
    assert f(0, 2, 8, hp=None, x=None, gl=None, lam=None, ho=None) == _lib.BLR_OK
    assert f(4, 0, 8, hp=FAKE, x=None, gl=None, ho=FAKE) == _lib.BLR_OK  # K = 0, in place: nothing to do


def test_step_validation(lib):
    f = lib.blr_step
    assert f(-1, 8, 0, 1.0, FAKE, FAKE, FAKE, FAKE, FAKE, None) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, 8, 3, 1.0, FAKE, FAKE, FAKE, FAKE, FAKE, None) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, 8, 0, 0.0, FAKE, FAKE, FAKE, FAKE, FAKE, None) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, 20, 0, 1.0, FAKE, FAKE, FAKE, FAKE, FAKE, None) == _lib.BLR_ERR_UNSUPPORTED
    assert f(0, 8, 0, 1.0, None, None, None, None, None, None) == _lib.BLR_OK
    assert f(4, 8, 0, 1.0, None, FAKE, FAKE, FAKE, FAKE, None) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, 8, 1, 1.0, FAKE, FAKE + 2, FAKE, FAKE, FAKE, None) == _lib.BLR_ERR_INVALID_ARG
    assert f(4, 8, 0, 1.0, FAKE, FAKE, FAKE, FAKE, FAKE + 4, None) == _lib.BLR_ERR_INVALID_ARG


def test_workspace_bytes(lib):
    wb = lambda *a: lib.blr_workspace_bytes(ctypes.byref(D(*a)))  # noqa: E731
    assert lib.blr_workspace_bytes(None) == 0
    assert wb(0, 10, 8) == 0 and wb(2, 0, 8) == 0 and wb(2, 10, 0) == 0
    assert wb(2, 10, 12) == 0 and wb(-1, 10, 8) == 0
    assert wb(1, 1, 8) > 0
    # it grows with the problem, stays a small fraction of it and ignores c
    small, large = wb(8, 1000, 64), wb(8, 4000, 64)
    assert large > small
    assert wb(8, 4000, 64, 0, 1.0) == wb(8, 4000, 64, 0, 3.0)
    for B, L, Dd, io in ((256, 200, 64, 0), (2048, 50, 64, 1), (64, 2048, 256, 0), (8, 2047, 512, 1)):
        n = B * L * Dd
        assert wb(B, L, Dd, io) < 0.5 * n + 64 * Dd + 4096, (B, L, Dd)
    # segmented problems keep the serial kernels' states, 8 bytes per channel
    # per segment of 128 steps or more, the chained forward's records (12 bytes
    # per channel per 128 steps) and the tiled backward records
    for B, L, Dd, io in ((8, 32768, 512, 1), (64, 2048, 64, 1), (3, 100000, 64, 1), (1, 65536, 8, 1)):
        n = B * L * Dd
        assert wb(B, L, Dd, io) < 0.95 * n + 24 * B * Dd + 64 * Dd + 4096, (B, L, Dd)


def test_scan_family(lib):
    """The kernel family follows the shape: 256 chains or more serial; fewer
    chains, bfloat16, L >= 2048 and 8 Mi elements or L >= 16384 segmented
    (tiled with row lengths); else tiled."""
    fam = lambda *a, lengths=0: lib.blr_scan_family(ctypes.byref(D(*a)), lengths)  # noqa: E731
    NONE, TILED, SERIAL, SEG = 0, 1, 2, 3
    assert lib.blr_scan_family(None, 0) == NONE
    assert fam(0, 10, 8) == NONE and fam(2, 0, 8) == NONE and fam(2, 10, 12) == NONE
    assert fam(256, 200, 64) == SERIAL          # 512 float32 chains
    assert fam(2048, 50, 64, 1) == SERIAL       # 2048 bfloat16 chains
    assert fam(64, 2048, 256) == SERIAL
    assert fam(255, 40000, 64, 1) == SEG        # 255 bfloat16 chains
    assert fam(256, 40000, 64, 1) == SERIAL
    assert fam(8, 32768, 512, 1) == SEG         # 64 bfloat16 chains
    assert fam(8, 32768, 512, 1, lengths=1) == TILED
    assert fam(8, 32768, 512, 0) == TILED       # float32: tiled
    assert fam(4, 50, 64, 1) == TILED
    assert fam(64, 2047, 64, 1) == TILED and fam(64, 2048, 64, 1) == SEG   # 8 Mi elements
    assert fam(4, 4096, 256, 1) == TILED        # 4 Mi elements, L < 16384
    assert fam(1, 16384, 64, 1) == SEG and fam(1, 16383, 64, 1) == TILED
    # a bfloat16 chain is 64 channels wide: (2, 4096) float32 rows make 256
    # chains, bfloat16 ones 128
    assert fam(2, 4096, 4096, 0) == SERIAL and fam(2, 4096, 4096, 1) == SEG


def test_status_strings(lib):
    for code in range(6):
        s = lib.blr_status_string(code)
        assert s and s.startswith(b"BLR_")
    assert b"unknown" in lib.blr_status_string(99)


def test_no_library_no_fallback(monkeypatch, tmp_path):
    """Without libblr.so every entry point raises: there is no CPU path."""
    import paper_2406_12580_gb300 as P
    monkeypatch.setattr(_lib, "_lib", None)
    monkeypatch.setattr(_lib, "library_path", lambda: str(tmp_path / "libblr.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        P.blr_workspace_bytes(D(2, 4, 8))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        P.blr_status_string(0)
