"""CPU: the seeded input generator (rounding, the Lambda initialisation, padding)."""
import numpy as np
import torch

from paper_2406_12580_gb300 import inputs as I


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    a = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 10,
                        np.array([0.0, -0.0, 1.0, -1.0, 3.0e38, 1e-40], np.float32)])
    # values exactly halfway between two bf16 numbers (ties to even)
    ties = (np.arange(1, 2000, dtype=np.uint32) << 16 | 0x8000).view(np.float32)
    a = np.concatenate([a, ties, -ties])
    bits = I.round_to_bf16(a)
    want = torch.from_numpy(a).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(bits, want)
    assert np.array_equal(I.bf16_bits_to_f32(bits), torch.from_numpy(a).to(torch.bfloat16).float().numpy())


def test_lambda_initialisation():
    # Sec. 3.2: exp(-softplus(Lambda)) uniform in [lo, hi]
    u = np.linspace(0.9, 0.999, 50)
    lam = I.lambda_from_decay(u)
    assert np.allclose(np.exp(-np.logaddexp(0.0, lam)), u, rtol=1e-13)
    inp = I.make_scan_inputs(I.scaled(I.CONFIGS[3], B=2, L=8))
    base = np.exp(-np.logaddexp(0.0, inp.lam.astype(np.float64)))
    assert base.min() >= 0.99 - 1e-6 and base.max() <= 0.9999 + 1e-6


def test_padding_and_determinism():
    cfg = I.scaled(I.CONFIGS[2], B=5)
    a = I.make_scan_inputs(cfg)
    b = I.make_scan_inputs(cfg)
    for name in ("x", "gl", "dh"):
        assert np.array_equal(getattr(a, name), getattr(b, name))
        assert np.array_equal(a.bits[name], b.bits[name])
    p = cfg.pad_rows
    assert p == 10
    assert not a.x[:, :p].any() and not a.gl[:, :p].any()
    assert a.x[:, p:].all() and a.dh[:, :p].any()
    # bf16 values round-trip exactly through their bit patterns
    assert np.array_equal(I.bf16_bits_to_f32(a.bits["x"]), a.x)
    assert a.gl.shape == (5, 50, 128) and a.x.dtype == np.float32


def test_step_inputs_shapes():
    cfg = I.StepConfig("t", B=7, D=16, io=I.BF16, seed=3)
    s = I.make_step_inputs(cfg)
    assert s.h_prev.shape == (7, 16) and s.gl.shape == (7, 32)
    assert s.bits["x"].dtype == np.uint16
