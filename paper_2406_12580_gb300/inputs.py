"""Seeded synthetic inputs for the BD-LRU scan, shared by the tests, the bench and the oracle.

This module holds no part of the method's arithmetic: it draws random numbers,
rounds them to the I/O dtype and lays them out. Both the CUDA path and the
oracle consume exactly the values produced here (the oracle upcasts them to
float64), so a parity test compares the two on identical inputs.

Workloads stand in for the paper's datasets (Sec. 4.1, Table "dataset"), which
are not available: only their shapes are used. L = 50 is the maximum length of
the Beauty / Sports / Steam runs and L = 200 that of ML-1M, the training batch
is 2048 and the embedding width 64 (Sec. 4.1, implementation details); XLong's
long histories (mean length 785.9) are scaled up in the long configurations.

The decay parameter Lambda follows the initialisation of Sec. 3.2: the base decay
exp(-softplus(Lambda)) is uniform in [lo, hi]. Writing u for that base decay,
exp(-softplus(Lambda)) = 1 / (1 + e^Lambda), so Lambda = log((1 - u) / u).

Draw order from one generator seeded with the configuration's seed:
Lambda uniforms (D), x (B*L*D), rho (B*L*D), iota (B*L*D), dh (B*L*D),
then the optional h0 / dh_last (B*D each). Zero left-padding is applied after
all draws, so it does not shift the stream.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import Optional

import numpy as np

F32 = "f32"
BF16 = "bf16"


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round to nearest, ties to even).

    Returns the uint16 bit patterns. Inputs are finite (no NaN handling)."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact upcast of bfloat16 bit patterns to float32."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


@dataclass(frozen=True)
class ScanConfig:
    """Shape, dtype and value recipe of one synthetic scan workload."""

    name: str
    B: int
    L: int
    D: int
    io: str = F32                      # I/O dtype of x, gate logits, dh, h, dx, dgl
    seed: int = 0
    x_std: float = 1.0
    gate_std: float = 1.0              # std of rho and iota (pre-activation logits)
    dh_std: float = 1.0
    decay: tuple = (0.9, 0.999)        # exp(-softplus(Lambda)) ~ U[lo, hi]
    pad_frac: float = 0.0              # leading fraction of each sequence set to zero rows
    fwd_only: bool = False
    random_h0: bool = False
    random_dh_last: bool = False
    c: float = 1.0
    gated: bool = False                # also draw z, the gated layer's merge input (Alg. 1)

    @property
    def elements(self) -> int:
        return self.B * self.L * self.D

    @property
    def pad_rows(self) -> int:
        return int(np.floor(self.pad_frac * self.L))


@dataclass(frozen=True)
class StepConfig:
    """Shape and value recipe of one recurrent-inference step workload."""

    name: str
    B: int
    D: int
    io: str = F32
    seed: int = 0
    decay: tuple = (0.99, 0.9999)
    c: float = 1.0

    @property
    def elements(self) -> int:
        return self.B * self.D


# The five workloads of the benchmark (the fifth adds a single-step run).
CONFIGS = {
    0: ScanConfig("fwd-only B=4 L=50 D=64 fp32", 4, 50, 64, F32, seed=0, fwd_only=True),
    1: ScanConfig("fwd+bwd B=256 L=200 D=64 fp32", 256, 200, 64, F32, seed=1),
    2: ScanConfig("train-shaped fwd+bwd B=2048 L=50 D=64 bf16, 20% left-padded", 2048, 50, 64,
                  BF16, seed=2, gate_std=0.5, pad_frac=0.2),
    3: ScanConfig("long-history fwd+bwd B=64 L=2048 D=256 fp32", 64, 2048, 256, F32, seed=3,
                  decay=(0.99, 0.9999)),
    4: ScanConfig("long-sequence fwd+bwd B=8 L=32768 D=512 bf16", 8, 32768, 512, BF16, seed=4,
                  decay=(0.99, 0.9999)),
}
STEP_CONFIG = StepConfig("recurrent step B=65536 D=64 fp32", 65536, 64, F32, seed=4)


@dataclass
class ScanInputs:
    """One workload's arrays. Float arrays hold values exactly representable in
    the I/O dtype; ``*_bits`` hold the bf16 bit patterns when io == bf16."""

    cfg: ScanConfig
    x: np.ndarray              # (B, L, D) float32
    gl: np.ndarray             # (B, L, 2D) float32: [..., :D] = rho, [..., D:] = iota
    lam: np.ndarray            # (D,) float32
    dh: Optional[np.ndarray]   # (B, L, D) float32 or None
    h0: Optional[np.ndarray]   # (B, D) float32 or None (zero state)
    dh_last: Optional[np.ndarray]  # (B, D) float32 or None
    bits: dict = field(default_factory=dict)
    z: Optional[np.ndarray] = None     # (B, L, D) float32 when cfg.gated (dh is then dy)

    def io_array(self, name: str) -> np.ndarray:
        """The array as the device sees it: float32, or uint16 bf16 bits."""
        if self.cfg.io == BF16:
            return self.bits[name]
        return getattr(self, name)


def lambda_from_decay(u: np.ndarray) -> np.ndarray:
    """Lambda with exp(-softplus(Lambda)) = u (the Sec. 3.2 initialisation)."""
    u = np.asarray(u, dtype=np.float64)
    return np.log((1.0 - u) / u)


def _normal(rng, n, std):
    v = rng.standard_normal(n, dtype=np.float32)
    if std != 1.0:
        v *= np.float32(std)
    return v


def _to_io(a: np.ndarray, io: str):
    if io == BF16:
        bits = round_to_bf16(a)
        return bf16_bits_to_f32(bits).reshape(a.shape), bits.reshape(a.shape)
    return np.ascontiguousarray(a, dtype=np.float32), None


def make_scan_inputs(cfg: ScanConfig) -> ScanInputs:
    """Draw one workload from ``cfg`` (deterministic in ``cfg.seed``)."""
    B, L, D = cfg.B, cfg.L, cfg.D
    rng = np.random.default_rng(cfg.seed)
    lo, hi = cfg.decay
    u = rng.uniform(lo, hi, size=D)
    lam = lambda_from_decay(u).astype(np.float32)
    n = B * L * D
    x = _normal(rng, n, cfg.x_std).reshape(B, L, D)
    rho = _normal(rng, n, cfg.gate_std).reshape(B, L, D)
    iota = _normal(rng, n, cfg.gate_std).reshape(B, L, D)
    dh = None if cfg.fwd_only else _normal(rng, n, cfg.dh_std).reshape(B, L, D)
    h0 = _normal(rng, B * D, 1.0).reshape(B, D) if cfg.random_h0 else None
    dh_last = _normal(rng, B * D, 1.0).reshape(B, D) if cfg.random_dh_last else None
    p = cfg.pad_rows
    if p > 0:
        x[:, :p, :] = 0.0
        rho[:, :p, :] = 0.0
        iota[:, :p, :] = 0.0
    gl = np.concatenate([rho, iota], axis=2)
    del rho, iota
    inp = ScanInputs(cfg, None, None, lam, None, h0, dh_last)
    bits = {}
    inp.x, bits["x"] = _to_io(x, cfg.io)
    del x
    inp.gl, bits["gl"] = _to_io(gl, cfg.io)
    del gl
    if dh is not None:
        inp.dh, bits["dh"] = _to_io(dh, cfg.io)
    if cfg.gated:  # a stream of its own, so the other arrays do not depend on it
        z = _normal(np.random.default_rng([cfg.seed, 2]), n, 1.0).reshape(B, L, D)
        inp.z, bits["z"] = _to_io(z, cfg.io)
    inp.bits = {k: v for k, v in bits.items() if v is not None}
    return inp


@dataclass
class StepInputs:
    cfg: StepConfig
    h_prev: np.ndarray   # (B, D) float32 (state is always fp32)
    x: np.ndarray        # (B, D) float32 values in the I/O dtype
    gl: np.ndarray       # (B, 2D)
    lam: np.ndarray      # (D,)
    bits: dict = field(default_factory=dict)

    def io_array(self, name: str) -> np.ndarray:
        if self.cfg.io == BF16:
            return self.bits[name]
        return getattr(self, name)


def make_step_inputs(cfg: StepConfig) -> StepInputs:
    """Draw one recurrent-step workload. Order: Lambda uniforms, h_prev, x, rho, iota.
    A second stream of the configuration seed is used so that it never
    coincides with the scan workload of the same seed."""
    rng = np.random.default_rng([cfg.seed, 1])
    B, D = cfg.B, cfg.D
    lo, hi = cfg.decay
    lam = lambda_from_decay(rng.uniform(lo, hi, size=D)).astype(np.float32)
    h_prev = _normal(rng, B * D, 1.0).reshape(B, D)
    x = _normal(rng, B * D, 1.0).reshape(B, D)
    rho = _normal(rng, B * D, 1.0).reshape(B, D)
    iota = _normal(rng, B * D, 1.0).reshape(B, D)
    gl = np.concatenate([rho, iota], axis=1)
    out = StepInputs(cfg, h_prev, None, None, lam)
    bits = {}
    out.x, bits["x"] = _to_io(x, cfg.io)
    out.gl, bits["gl"] = _to_io(gl, cfg.io)
    out.bits = {k: v for k, v in bits.items() if v is not None}
    return out


def scaled(cfg: ScanConfig, **changes) -> ScanConfig:
    """A copy of ``cfg`` with some fields replaced (e.g. a smaller B for a test)."""
    return replace(cfg, **changes)
