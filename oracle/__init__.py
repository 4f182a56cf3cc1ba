"""Float64 CPU oracle for the BD-LRU scan (RecBLR, arXiv 2406.12580, Sec. 3.2).

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import this package. The product path (the
CUDA library and its Python binding) never imports, links or runs it.

The arithmetic lives in ``blr_oracle.c`` (plain C99, float64, serial per
channel, optional OpenMP across independent channels). This module only builds
that file with gcc and marshals numpy arrays to it.

Functions and the passages they follow:
  gates(gl, lam, c)                 -> alpha_t, beta_t       Sec. 3.2 (gate and decay equations)
  fwd(x, gl, lam, h0, c)            -> h, h_last             Sec. 3.2, Eq. linrnn
  bwd(dh, x, gl, lam, h0, dh_last)  -> dx, dgl, dlam, dh0    chain rule of Sec. 3.2 (not printed in the paper)
  step(h_prev, x, gl, lam, c)       -> h_t                   Sec. 1 / Sec. 4.3 (recurrent inference)
  steps(h_prev, x, gl, lam, c)      -> h_seq, h_out         K recurrent steps per row (step, repeated)
  fwd_varlen / bwd_varlen(lengths, ...)                     per-row lengths: row b is its last lengths[b]
                                                            steps (Sec. 3.3's left padding, not read)
  fwd_gated(x, gl, lam, z, h0, c)   -> y = h SiLU(z), h_last  Alg. 1 (the scan, then the merge H_y (x) SiLU(H_z))
  bwd_gated(dy, x, gl, lam, z, ...) -> dx, dgl, dlam, dh0, dz  chain rule through the merge, then bwd

Every function is pinned by the CPU tests in ``tests/test_oracle_pins.py``
(closed forms, special cases, brute force, the paper's two-tree scan,
finite differences); none is left unpinned.
"""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess
import tempfile
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "blr_oracle.c")
LIBRARY = os.path.join(_HERE, "libblr_oracle.so")

# -ffp-contract=off keeps a*b+c as two roundings on every host (aarch64 gcc
# would otherwise fuse them), so the oracle gives the same bits on x86 and Arm.
CFLAGS = ["-O2", "-std=c99", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]

_lock = threading.Lock()


def build(source: str = SOURCE, output: str = LIBRARY, extra_flags=(), openmp: bool = True) -> str:
    """Compile the oracle C source into a shared library (atomic rename)."""
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        raise RuntimeError("no C compiler found to build the oracle")
    flags = list(CFLAGS) + list(extra_flags)
    if openmp:
        flags.append("-fopenmp")
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=os.path.dirname(output) or ".")
    os.close(fd)
    try:
        subprocess.run([cc, *flags, source, "-o", tmp, "-lm"], check=True,
                       stdout=subprocess.PIPE, stderr=subprocess.STDOUT)
        os.replace(tmp, output)
    finally:
        if os.path.exists(tmp):
            os.unlink(tmp)
    return output


def _stale(lib: str, src: str) -> bool:
    return (not os.path.exists(lib)) or os.path.getmtime(lib) < os.path.getmtime(src)


_P = ctypes.POINTER(ctypes.c_double)
_I64 = ctypes.c_int64


def _ptr(a):
    return None if a is None else a.ctypes.data_as(_P)


def _f64(a, shape=None):
    if a is None:
        return None
    a = np.ascontiguousarray(a, dtype=np.float64)
    if shape is not None and a.shape != tuple(shape):
        raise ValueError(f"expected shape {tuple(shape)}, got {a.shape}")
    return a


class Oracle:
    """ctypes front end of one built oracle library (see module docstring)."""

    def __init__(self, path: str):
        self.path = path
        lib = ctypes.CDLL(path)
        lib.blr_oracle_gates.argtypes = [_I64, _I64, _I64, ctypes.c_double, _P, _P, _P, _P]
        lib.blr_oracle_fwd.argtypes = [_I64, _I64, _I64, ctypes.c_double, _P, _P, _P, _P, _P, _P,
                                       ctypes.c_int]
        lib.blr_oracle_bwd.argtypes = [_I64, _I64, _I64, ctypes.c_double, _P, _P, _P, _P, _P, _P,
                                       _P, _P, _P, _P, ctypes.c_int]
        lib.blr_oracle_step.argtypes = [_I64, _I64, ctypes.c_double, _P, _P, _P, _P, _P]
        lib.blr_oracle_merge.argtypes = [_I64, _P, _P, _P]
        lib.blr_oracle_merge_bwd.argtypes = [_I64, _P, _P, _P, _P, _P]
        lib.blr_oracle_has_openmp.restype = ctypes.c_int
        for f in ("blr_oracle_gates", "blr_oracle_fwd", "blr_oracle_bwd", "blr_oracle_step",
                  "blr_oracle_merge", "blr_oracle_merge_bwd"):
            getattr(lib, f).restype = None
        self._lib = lib
        self.has_openmp = bool(lib.blr_oracle_has_openmp())

    @staticmethod
    def _dims(x, gl, lam):
        B, L, D = x.shape
        if gl.shape != (B, L, 2 * D) or lam.shape != (D,):
            raise ValueError(f"shape mismatch: x {x.shape}, gl {gl.shape}, lam {lam.shape}")
        return B, L, D

    def gates(self, gl, lam, c: float = 1.0):
        gl, lam = _f64(gl), _f64(lam)
        B, L, D2 = gl.shape
        D = D2 // 2
        alpha = np.empty((B, L, D))
        beta = np.empty((B, L, D))
        self._lib.blr_oracle_gates(B, L, D, c, _ptr(gl), _ptr(lam), _ptr(alpha), _ptr(beta))
        return alpha, beta

    def fwd(self, x, gl, lam, h0=None, c: float = 1.0, threads: int = 1):
        x, gl, lam = _f64(x), _f64(gl), _f64(lam)
        B, L, D = self._dims(x, gl, lam)
        h0 = _f64(h0, (B, D))
        h = np.empty((B, L, D))
        h_last = np.empty((B, D))
        self._lib.blr_oracle_fwd(B, L, D, c, _ptr(x), _ptr(gl), _ptr(lam), _ptr(h0), _ptr(h),
                                 _ptr(h_last), threads)
        return h, h_last

    def bwd(self, dh, x, gl, lam, h0=None, dh_last=None, c: float = 1.0, threads: int = 1):
        x, gl, lam = _f64(x), _f64(gl), _f64(lam)
        B, L, D = self._dims(x, gl, lam)
        dh = _f64(dh, (B, L, D))
        h0 = _f64(h0, (B, D))
        dh_last = _f64(dh_last, (B, D))
        dx = np.empty((B, L, D))
        dgl = np.empty((B, L, 2 * D))
        dlam = np.empty((D,))
        dh0 = np.empty((B, D))
        self._lib.blr_oracle_bwd(B, L, D, c, _ptr(dh), _ptr(dh_last), _ptr(x), _ptr(gl),
                                 _ptr(lam), _ptr(h0), _ptr(dx), _ptr(dgl), _ptr(dlam),
                                 _ptr(dh0), threads)
        return dx, dgl, dlam, dh0

    def step(self, h_prev, x, gl, lam, c: float = 1.0):
        x, lam = _f64(x), _f64(lam)
        B, D = x.shape
        h_prev = _f64(h_prev, (B, D))
        gl = _f64(gl, (B, 2 * D))
        lam = _f64(lam, (D,))
        h_t = np.empty((B, D))
        self._lib.blr_oracle_step(B, D, c, _ptr(h_prev), _ptr(x), _ptr(gl), _ptr(lam), _ptr(h_t))
        return h_t

    def steps(self, h_prev, x, gl, lam, c: float = 1.0):
        """K consecutive recurrent steps of every row: x (B, K, D), gl (B, K, 2D).
        Returns (h_seq (B, K, D), h_out (B, D)); one call of step per step."""
        x, gl = _f64(x), _f64(gl)
        B, K, D = x.shape
        h = _f64(h_prev, (B, D))
        h_seq = np.empty((B, K, D))
        for j in range(K):
            h = self.step(h, x[:, j], gl[:, j], lam, c=c)
            h_seq[:, j] = h
        return h_seq, h

    def fwd_varlen(self, lengths, x, gl, lam, h0=None, c: float = 1.0, threads: int = 1):
        """Row b is a sequence of its last lengths[b] steps (rows [L - len, L));
        the rows before it are not part of it. Returns (h, h_last) with h NaN on
        those rows (nothing is computed there)."""
        x, gl, lam = _f64(x), _f64(gl), _f64(lam)
        B, L, D = self._dims(x, gl, lam)
        h = np.full((B, L, D), np.nan)
        h_last = np.empty((B, D))
        for b in range(B):
            t0 = L - int(lengths[b])
            hb0 = None if h0 is None else _f64(h0)[b:b + 1]
            if t0 == L:
                h_last[b] = 0.0 if hb0 is None else hb0[0]
                continue
            hb, hl = self.fwd(x[b:b + 1, t0:], gl[b:b + 1, t0:], lam, hb0, c=c, threads=threads)
            h[b, t0:] = hb[0]
            h_last[b] = hl[0]
        return h, h_last

    def bwd_varlen(self, lengths, dh, x, gl, lam, h0=None, dh_last=None, c: float = 1.0,
                   threads: int = 1):
        """Backward of fwd_varlen: (dx, dgl, dlam, dh0), dx and dgl NaN on the rows
        before each sequence; dh there is not read."""
        x, gl, lam = _f64(x), _f64(gl), _f64(lam)
        B, L, D = self._dims(x, gl, lam)
        dh = _f64(dh, (B, L, D))
        dx = np.full((B, L, D), np.nan)
        dgl = np.full((B, L, 2 * D), np.nan)
        dlam = np.zeros(D)
        dh0 = np.empty((B, D))
        for b in range(B):
            t0 = L - int(lengths[b])
            dl = np.zeros(D) if dh_last is None else _f64(dh_last)[b]
            if t0 == L:
                dh0[b] = dl
                continue
            hb0 = None if h0 is None else _f64(h0)[b:b + 1]
            g = self.bwd(dh[b:b + 1, t0:], x[b:b + 1, t0:], gl[b:b + 1, t0:], lam, hb0,
                         dl[None], c=c, threads=threads)
            dx[b, t0:], dgl[b, t0:] = g[0][0], g[1][0]
            dlam += g[2]
            dh0[b] = g[3][0]
        return dx, dgl, dlam, dh0

    def merge(self, h, z):
        """y = h SiLU(z), elementwise (Alg. 1, the merge of the two branches)."""
        h = _f64(h)
        z = _f64(z, h.shape)
        y = np.empty(h.shape)
        self._lib.blr_oracle_merge(h.size, _ptr(h), _ptr(z), _ptr(y))
        return y

    def merge_bwd(self, dy, h, z):
        """(dh, dz) of the merge for the upstream gradient dy."""
        h = _f64(h)
        dy, z = _f64(dy, h.shape), _f64(z, h.shape)
        dh, dz = np.empty(h.shape), np.empty(h.shape)
        self._lib.blr_oracle_merge_bwd(h.size, _ptr(dy), _ptr(h), _ptr(z), _ptr(dh), _ptr(dz))
        return dh, dz

    def fwd_gated(self, x, gl, lam, z, h0=None, c: float = 1.0, threads: int = 1):
        """The scan followed by the merge: (y, h_last), y = h SiLU(z)."""
        h, h_last = self.fwd(x, gl, lam, h0, c=c, threads=threads)
        return self.merge(h, z), h_last

    def bwd_gated(self, dy, x, gl, lam, z, h0=None, dh_last=None, c: float = 1.0, threads: int = 1):
        """Backward of fwd_gated for the loss sum dy y + sum dh_last h_last:
        (dx, dgl, dlam, dh0, dz)."""
        h, _ = self.fwd(x, gl, lam, h0, c=c, threads=threads)
        dh, dz = self.merge_bwd(dy, h, z)
        dx, dgl, dlam, dh0 = self.bwd(dh, x, gl, lam, h0, dh_last, c=c, threads=threads)
        return dx, dgl, dlam, dh0, dz


_default = None


def load() -> Oracle:
    """The oracle built from ``blr_oracle.c`` (rebuilt when the source is newer)."""
    global _default
    with _lock:
        if _default is None:
            if _stale(LIBRARY, SOURCE):
                build()
            _default = Oracle(LIBRARY)
        return _default
