"""Checks that pin the float64 oracle to facts other than itself.

Each ``pin_*`` function takes an ``oracle.Oracle`` and raises AssertionError when
the oracle disagrees with something the paper or mathematics fixes:

  * hand-worked values at inputs where every gate has a closed form (golden fixture);
  * the geometric-sum closed form of a constant-gate recurrence;
  * the degenerate decays alpha -> 0 (h_t = i_t x_t) and alpha -> 1 (h frozen);
  * linearity in (x, h0) for fixed gates;
  * the O(L^2) unrolled sum, with gates from library primitives (scipy's expit,
    numpy's logaddexp), on tiny inputs;
  * the paper's two-tree parallel scan (Sec. 3.3, Fig. "scan") at T = 8;
  * zero left-padding invariance (Sec. 3.3, embedding padding), and per-row
    lengths against the zero-padded scan;
  * split / resume of the state;
  * the stability bound implied by alpha, beta in [0, 1] (Sec. 3.2);
  * central finite differences of every gradient, linearity of the gradient in
    dh, and consistency of the single step with a length-1 scan, of K steps
    with a length-K scan and with the closed form of constant gates;
  * for the merge of the gated layer (Alg. 1, y = h SiLU(z)): SiLU's values and
    slope at 0 and its limits z -> +-inf, the reduction to the plain scan at
    the z where SiLU(z) = 1 (found by root finding on scipy's expit), and
    central finite differences of every gradient through the merge.

They are plain functions (not tests) so that ``test_oracle_mutants.py`` can run
the same set against oracle builds with a planted mistake and show that each
mistake is caught.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np
from scipy.special import expit

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                      "bdlru_worked_example.json")


def _ev(expr: str) -> float:
    return float(eval(expr, {"__builtins__": {}}, {"sqrt": math.sqrt, "log": math.log}))


def _rel(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    scale = max(np.max(np.abs(b)), 1e-300)
    return float(np.max(np.abs(a - b)) / scale)


def _rand_problem(rng, B, L, D, decay=(0.5, 0.99), gate_std=1.0):
    u = rng.uniform(*decay, size=D)
    lam = np.log((1 - u) / u)
    x = rng.standard_normal((B, L, D))
    gl = rng.standard_normal((B, L, 2 * D)) * gate_std
    return x, gl, lam


def _lib_gates(gl, lam, c):
    """alpha, beta from library primitives (numpy logaddexp, scipy expit)."""
    D = lam.shape[0]
    s = np.logaddexp(0.0, lam)
    r = expit(gl[..., :D])
    i = expit(gl[..., D:])
    alpha = np.exp(-c * s * r)
    beta = np.sqrt(1.0 - alpha ** 2) * i
    return alpha, beta


# --------------------------------------------------------------------- forward


def pin_golden_forward(orc):
    with open(GOLDEN) as f:
        cases = json.load(f)["forward"]
    for case in cases:
        L = len(case["x"])
        x = np.array([_ev(v) for v in case["x"]]).reshape(1, L, 1)
        rho = [_ev(v) for v in case["rho"]]
        iota = [_ev(v) for v in case["iota"]]
        gl = np.array([[r, i] for r, i in zip(rho, iota)]).reshape(1, L, 2)
        lam = np.array([_ev(case["lambda"])])
        h0 = np.array([[_ev(case["h0"])]])
        h, h_last = orc.fwd(x, gl, lam, h0, c=case["c"])
        want = np.array([_ev(v) for v in case["h"]])
        assert np.allclose(h.ravel(), want, rtol=1e-13, atol=1e-15), (case["name"], h.ravel(), want)
        assert h_last[0, 0] == h[0, -1, 0]
        alpha, beta = orc.gates(gl, lam, c=case["c"])
        assert np.allclose(alpha, _ev(case["alpha"]), rtol=1e-14), case["name"]
        assert np.allclose(beta, _ev(case["beta"]), rtol=1e-14), case["name"]


def pin_geometric_closed_form(orc):
    # c = 2, Lambda = 0, rho = iota = 0 gives alpha = 1/2 and beta = sqrt(3)/4 exactly,
    # so with constant x the state is h_t = 2^-t h0 + x beta (1 - 2^-t) / (1 - 1/2).
    rng = np.random.default_rng(11)
    B, L, D = 2, 40, 3
    x0 = rng.standard_normal((B, 1, D))
    x = np.repeat(x0, L, axis=1)
    gl = np.zeros((B, L, 2 * D))
    lam = np.zeros(D)
    h0 = rng.standard_normal((B, D))
    h, _ = orc.fwd(x, gl, lam, h0, c=2.0)
    t = np.arange(1, L + 1).reshape(1, L, 1)
    want = 0.5 ** t * h0[:, None, :] + x0 * (math.sqrt(3) / 4) * (1 - 0.5 ** t) / 0.5
    assert _rel(h, want) < 1e-13
    # General constant gates per channel (gates from library primitives):
    rho = rng.standard_normal((1, 1, D)) * 2
    iota = rng.standard_normal((1, 1, D)) * 2
    lam = rng.standard_normal(D)
    gl = np.concatenate([np.broadcast_to(rho, (B, L, D)), np.broadcast_to(iota, (B, L, D))], 2)
    a, bt = _lib_gates(gl[:1, :1], lam, 1.0)
    h, _ = orc.fwd(x, gl, lam, h0, c=1.0)
    want = a ** t * h0[:, None, :] + bt * x0 * (1 - a ** t) / (1 - a)
    assert _rel(h, want) < 1e-12


def pin_alpha_zero(orc):
    # Lambda = 1000 and rho = 20: alpha = exp(-1000 r) underflows to 0, so h_t = i_t x_t.
    rng = np.random.default_rng(12)
    B, L, D = 2, 9, 4
    x = rng.standard_normal((B, L, D))
    iota = rng.standard_normal((B, L, D)) * 3
    gl = np.concatenate([np.full((B, L, D), 20.0), iota], axis=2)
    lam = np.full(D, 1000.0)
    h0 = rng.standard_normal((B, D))
    h, _ = orc.fwd(x, gl, lam, h0)
    assert _rel(h, expit(iota) * x) < 1e-15


def pin_alpha_one(orc):
    # Lambda = -50: softplus = 1.9e-22, alpha rounds to 1 and beta to 0: h stays h0.
    rng = np.random.default_rng(13)
    B, L, D = 2, 17, 3
    gl = rng.standard_normal((B, L, 2 * D))
    lam = np.full(D, -50.0)
    h0 = rng.standard_normal((B, D))
    for x in (np.zeros((B, L, D)), rng.standard_normal((B, L, D))):
        h, h_last = orc.fwd(x, gl, lam, h0)
        assert np.array_equal(h, np.broadcast_to(h0[:, None, :], h.shape))
        assert np.array_equal(h_last, h0)


def pin_linearity(orc):
    rng = np.random.default_rng(14)
    B, L, D = 3, 11, 5
    x1, gl, lam = _rand_problem(rng, B, L, D)
    x2 = rng.standard_normal((B, L, D))
    h01, h02 = rng.standard_normal((B, D)), rng.standard_normal((B, D))
    a, b = 0.7, -1.3
    h1, _ = orc.fwd(x1, gl, lam, h01)
    h2, _ = orc.fwd(x2, gl, lam, h02)
    h12, _ = orc.fwd(a * x1 + b * x2, gl, lam, a * h01 + b * h02)
    assert _rel(h12, a * h1 + b * h2) < 1e-13


def pin_bruteforce(orc):
    # h_t = sum_k (prod_{k<j<=t} alpha_j) beta_k x_k + (prod_{j<=t} alpha_j) h0
    rng = np.random.default_rng(15)
    B, L, D = 2, 7, 3
    c = 1.7
    x, gl, lam = _rand_problem(rng, B, L, D, decay=(0.3, 0.95))
    h0 = rng.standard_normal((B, D))
    alpha, beta = _lib_gates(gl, lam, c)
    want = np.zeros((B, L, D))
    for b in range(B):
        for d in range(D):
            for t in range(L):
                acc = np.prod(alpha[b, : t + 1, d]) * h0[b, d]
                for k in range(t + 1):
                    acc += np.prod(alpha[b, k + 1: t + 1, d]) * beta[b, k, d] * x[b, k, d]
                want[b, t, d] = acc
    h, _ = orc.fwd(x, gl, lam, h0, c=c)
    assert _rel(h, want) < 1e-13
    a2, b2 = orc.gates(gl, lam, c=c)
    assert _rel(a2, alpha) < 1e-14 and _rel(b2, beta) < 1e-14


def _compose(later, earlier):
    # (a2, b2) . (a1, b1) = (a2 a1, a2 b1 + b2)  (Sec. 3.3, the operator of the scan)
    return (later[0] * earlier[0], later[0] * earlier[1] + later[1])


def _two_tree_scan(c):
    """The paper's two-tree scan (Sec. 3.3, Fig. "scan") for a power-of-two T.

    Tree1 leaves hold c_T ... c_1 left to right; an up-sweep sets every inner
    node to Tree1[left] . Tree1[right]. Tree2's root is the identity; the
    down-sweep sets Tree2[right] = Tree2[v] and Tree2[left] = Tree1[right] . Tree2[v].
    Tree2's leaf above c_t then holds c_{t-1} . ... . c_1, and h_t = c_t . that."""
    T = len(c)
    assert T & (T - 1) == 0
    ident = (1.0, 0.0)
    leaves = list(reversed(c))           # leaf j (left to right) holds c_{T-j}
    tree1 = [None] * (2 * T)
    for j in range(T):
        tree1[T + j] = leaves[j]
    for v in range(T - 1, 0, -1):        # up-sweep (node v has children 2v, 2v+1)
        tree1[v] = _compose(tree1[2 * v], tree1[2 * v + 1])
    tree2 = [None] * (2 * T)
    tree2[1] = ident
    for v in range(1, T):                # down-sweep, parents before children
        tree2[2 * v + 1] = tree2[v]
        tree2[2 * v] = _compose(tree1[2 * v + 1], tree2[v])
    out = [None] * T
    for j in range(T):
        t = T - 1 - j                    # 0-based time index of this leaf
        out[t] = _compose(tree1[T + j], tree2[T + j])[1]
    return out


def pin_two_tree_scan(orc):
    rng = np.random.default_rng(16)
    B, L, D = 2, 8, 3
    x, gl, lam = _rand_problem(rng, B, L, D)
    alpha, beta = orc.gates(gl, lam)
    h, _ = orc.fwd(x, gl, lam, None)
    for b in range(B):
        for d in range(D):
            c = [(alpha[b, t, d], beta[b, t, d] * x[b, t, d]) for t in range(L)]
            got = _two_tree_scan(c)
            assert _rel(h[b, :, d], got) < 1e-13


def pin_left_padding(orc):
    # Zero rows prepended (any logits) leave the real rows unchanged from h0 = 0.
    rng = np.random.default_rng(17)
    B, L, D, P = 2, 13, 4, 19
    x, gl, lam = _rand_problem(rng, B, L, D)
    pad_gl = rng.standard_normal((B, P, 2 * D)) * 4
    xp = np.concatenate([np.zeros((B, P, D)), x], axis=1)
    glp = np.concatenate([pad_gl, gl], axis=1)
    h, hl = orc.fwd(x, gl, lam, None)
    hp, hlp = orc.fwd(xp, glp, lam, None)
    assert np.array_equal(hp[:, P:], h) and np.array_equal(hlp, hl)
    assert np.array_equal(hp[:, :P], np.zeros((B, P, D)))


def pin_split_resume(orc):
    rng = np.random.default_rng(18)
    B, L, D, k = 2, 23, 3, 9
    x, gl, lam = _rand_problem(rng, B, L, D)
    h0 = rng.standard_normal((B, D))
    h, hl = orc.fwd(x, gl, lam, h0)
    ha, hla = orc.fwd(x[:, :k], gl[:, :k], lam, h0)
    hb, hlb = orc.fwd(x[:, k:], gl[:, k:], lam, hla)
    assert np.array_equal(np.concatenate([ha, hb], axis=1), h)
    assert np.array_equal(hlb, hl)


def pin_bound(orc):
    # alpha_t <= abar < 1, h0 = 0 and |beta x| <= |x|: |h_t| <= max|x| / (1 - abar).
    rng = np.random.default_rng(19)
    B, L, D = 4, 300, 6
    x, gl, lam = _rand_problem(rng, B, L, D, decay=(0.8, 0.95))
    alpha, beta = _lib_gates(gl, lam, 1.0)
    abar = alpha.max()
    h, _ = orc.fwd(x, gl, lam, None)
    assert np.all(np.abs(h) <= np.abs(x).max() / (1 - abar) + 1e-12)
    assert np.all((alpha >= 0) & (alpha <= 1) & (beta >= 0) & (beta <= 1))


# -------------------------------------------------------------------- backward


def pin_golden_backward(orc):
    with open(GOLDEN) as f:
        case = json.load(f)["backward"][0]
    x = np.array([[[_ev(case["x"])]]])
    gl = np.array([[[_ev(case["rho"]), _ev(case["iota"])]]])
    lam = np.array([_ev(case["lambda"])])
    h0 = np.array([[_ev(case["h0"])]])
    dh = np.array([[[_ev(case["dh"])]]])
    dx, dgl, dlam, dh0 = orc.bwd(dh, x, gl, lam, h0, None, c=case["c"])
    for got, key in ((dx[0, 0, 0], "dx"), (dgl[0, 0, 0], "drho"), (dgl[0, 0, 1], "diota"),
                     (dlam[0], "dlambda"), (dh0[0, 0], "dh0")):
        want = _ev(case[key])
        assert abs(got - want) <= 1e-14 * max(1.0, abs(want)), (key, got, want)


def _loss(orc, x, gl, lam, h0, dh, dh_last, c):
    h, hl = orc.fwd(x, gl, lam, h0, c=c)
    return float(np.sum(dh * h) + np.sum(dh_last * hl))


def pin_finite_differences(orc):
    rng = np.random.default_rng(20)
    B, L, D, c = 2, 6, 3, 1.3
    x, gl, lam = _rand_problem(rng, B, L, D, decay=(0.6, 0.97))
    h0 = rng.standard_normal((B, D))
    dh = rng.standard_normal((B, L, D))
    dh_last = rng.standard_normal((B, D))
    dx, dgl, dlam, dh0 = orc.bwd(dh, x, gl, lam, h0, dh_last, c=c)
    eps = 1e-6

    def fd(arr, setter):
        out = np.empty_like(arr)
        for idx in np.ndindex(arr.shape):
            p = arr.copy(); p[idx] += eps
            m = arr.copy(); m[idx] -= eps
            out[idx] = (setter(p) - setter(m)) / (2 * eps)
        return out

    fx = fd(x, lambda v: _loss(orc, v, gl, lam, h0, dh, dh_last, c))
    fgl = fd(gl, lambda v: _loss(orc, x, v, lam, h0, dh, dh_last, c))
    flam = fd(lam, lambda v: _loss(orc, x, gl, v, h0, dh, dh_last, c))
    fh0 = fd(h0, lambda v: _loss(orc, x, gl, lam, v, dh, dh_last, c))
    for got, want, name in ((dx, fx, "dx"), (dgl, fgl, "dgl"), (dlam, flam, "dlambda"),
                            (dh0, fh0, "dh0")):
        assert _rel(got, want) < 1e-6, (name, _rel(got, want))


def pin_gradient_linearity(orc):
    rng = np.random.default_rng(21)
    B, L, D = 2, 10, 4
    x, gl, lam = _rand_problem(rng, B, L, D)
    h0 = rng.standard_normal((B, D))
    d1, d2 = rng.standard_normal((B, L, D)), rng.standard_normal((B, L, D))
    l1, l2 = rng.standard_normal((B, D)), rng.standard_normal((B, D))
    a, b = -0.4, 2.5
    g1 = orc.bwd(d1, x, gl, lam, h0, l1)
    g2 = orc.bwd(d2, x, gl, lam, h0, l2)
    g12 = orc.bwd(a * d1 + b * d2, x, gl, lam, h0, a * l1 + b * l2)
    for u, v, w in zip(g1, g2, g12):
        assert _rel(w, a * u + b * v) < 1e-12


def pin_step(orc):
    rng = np.random.default_rng(22)
    B, D = 5, 6
    x, gl, lam = _rand_problem(rng, B, 1, D)
    h_prev = rng.standard_normal((B, D))
    h, _ = orc.fwd(x, gl, lam, h_prev, c=1.5)
    ht = orc.step(h_prev, x[:, 0], gl[:, 0], lam, c=1.5)
    assert np.array_equal(ht, h[:, 0])
    # closed form: c = 2, Lambda = rho = iota = 0 -> h = h_prev / 2 + sqrt(3)/4 x
    ht = orc.step(h_prev, x[:, 0], np.zeros((B, 2 * D)), np.zeros(D), c=2.0)
    assert _rel(ht, 0.5 * h_prev + math.sqrt(3) / 4 * x[:, 0]) < 1e-15


def pin_steps(orc):
    rng = np.random.default_rng(26)
    B, K, D = 4, 7, 5
    x, gl, lam = _rand_problem(rng, B, K, D)
    h_prev = rng.standard_normal((B, D))
    h_seq, h_out = orc.steps(h_prev, x, gl, lam, c=1.3)
    h, hl = orc.fwd(x, gl, lam, h_prev, c=1.3)  # K steps are a length-K scan from h_prev
    assert np.array_equal(h_seq, h) and np.array_equal(h_out, hl)
    # closed form: c = 2, Lambda = rho = iota = 0 -> alpha = 1/2, beta = sqrt(3)/4 every step
    _, h_out = orc.steps(h_prev, x, np.zeros((B, K, 2 * D)), np.zeros(D), c=2.0)
    want = 0.5 ** K * h_prev + sum(0.5 ** (K - 1 - j) * math.sqrt(3) / 4 * x[:, j] for j in range(K))
    assert _rel(h_out, want) < 1e-14


def pin_varlen_is_zero_left_padding(orc):
    # Sec. 3.3: sequences left-padded with zero rows scan to the same states (h0
    # = 0); so a per-row length that skips the padding must give the padded
    # scan's values on the real rows, and the same gate and Lambda gradients
    # when dh is zero on the padding. dh0 differs by the padding's decay.
    rng = np.random.default_rng(27)
    B, L, D, c = 4, 12, 3, 1.2
    x, gl, lam = _rand_problem(rng, B, L, D)
    lengths = np.array([12, 7, 1, 0])
    dh = rng.standard_normal((B, L, D))
    dh_last = rng.standard_normal((B, D))
    for b, n in enumerate(lengths):
        x[b, :L - n] = 0.0
        gl[b, :L - n] = 0.0
        dh[b, :L - n] = 0.0
    h, hl = orc.fwd(x, gl, lam, None, c=c)
    hv, hlv = orc.fwd_varlen(lengths, x, gl, lam, None, c=c)
    real = ~np.isnan(hv)
    assert np.array_equal(real, np.broadcast_to((np.arange(L)[None, :, None] >= (L - lengths)[:, None, None]), real.shape))
    assert _rel(hv[real], h[real]) < 1e-14 and _rel(hlv, hl) < 1e-14
    dx, dgl, dlam, dh0 = orc.bwd(dh, x, gl, lam, None, dh_last, c=c)
    dxv, dglv, dlamv, dh0v = orc.bwd_varlen(lengths, dh, x, gl, lam, None, dh_last, c=c)
    assert _rel(dxv[real], dx[real]) < 1e-13
    real2 = np.concatenate([real, real], axis=2)
    assert _rel(dglv[real2], dgl[real2]) < 1e-13
    assert _rel(dlamv, dlam) < 1e-13
    # padding rows have x = rho = iota = 0: alpha = exp(c * k / 2) each, k = -softplus
    apad = np.exp(-c * np.logaddexp(0.0, lam) * 0.5)
    for b, n in enumerate(lengths):
        assert _rel(dh0[b], dh0v[b] * apad ** (L - n)) < 1e-13


def pin_varlen_full_and_empty(orc):
    rng = np.random.default_rng(28)
    B, L, D = 3, 9, 4
    x, gl, lam = _rand_problem(rng, B, L, D)
    h0 = rng.standard_normal((B, D))
    dh = rng.standard_normal((B, L, D))
    full = np.full(B, L)
    h, hl = orc.fwd(x, gl, lam, h0)
    hv, hlv = orc.fwd_varlen(full, x, gl, lam, h0)
    assert np.array_equal(h, hv) and np.array_equal(hl, hlv)
    g = orc.bwd(dh, x, gl, lam, h0, None)
    gv = orc.bwd_varlen(full, dh, x, gl, lam, h0, None)
    for a_, b_ in zip(g, gv):
        assert _rel(b_, a_) < 1e-14
    # empty sequences: the state is h0, its gradient dh_last, nothing else moves
    dh_last = rng.standard_normal((B, D))
    _, hl0 = orc.fwd_varlen(np.zeros(B, dtype=int), x, gl, lam, h0)
    assert np.array_equal(hl0, h0)
    _, _, dlam0, dh00 = orc.bwd_varlen(np.zeros(B, dtype=int), dh, x, gl, lam, h0, dh_last)
    assert np.array_equal(dh00, dh_last) and np.array_equal(dlam0, np.zeros(D))


# ----------------------------------------------------- the gated layer's merge


def pin_merge_limits(orc):
    rng = np.random.default_rng(23)
    h = rng.standard_normal((3, 7, 4))
    dy = rng.standard_normal(h.shape)
    zeros = np.zeros_like(h)
    # SiLU(0) = 0 and SiLU'(0) = 1/2
    assert np.array_equal(orc.merge(h, zeros), zeros)
    dh, dz = orc.merge_bwd(dy, h, zeros)
    assert np.array_equal(dh, zeros)
    assert _rel(dz, 0.5 * dy * h) < 1e-15
    # z -> +inf: SiLU(z) / z -> 1 and SiLU'(z) -> 1; z -> -inf: both -> 0
    big = np.full_like(h, 40.0)
    assert _rel(orc.merge(h, big), 40.0 * h) < 1e-15
    dh, dz = orc.merge_bwd(dy, h, big)
    assert _rel(dh, 40.0 * dy) < 1e-15 and _rel(dz, dy * h) < 1e-15
    y = orc.merge(h, -big)
    assert np.max(np.abs(y)) <= 40.0 * math.exp(-40.0) * np.max(np.abs(h))
    dh, dz = orc.merge_bwd(dy, h, -big)
    assert np.max(np.abs(dz)) <= 41.0 * 40.0 * math.exp(-40.0) * np.max(np.abs(dy * h))


def pin_merge_unit_gate(orc):
    from scipy.optimize import brentq
    z1 = brentq(lambda z: z * expit(z) - 1.0, 0.0, 5.0, xtol=1e-15, rtol=1e-15)  # SiLU(z1) = 1
    rng = np.random.default_rng(24)
    B, L, D, c = 2, 9, 3, 1.7
    x, gl, lam = _rand_problem(rng, B, L, D)
    h0 = rng.standard_normal((B, D))
    dy = rng.standard_normal((B, L, D))
    dh_last = rng.standard_normal((B, D))
    z = np.full((B, L, D), z1)
    y, yl = orc.fwd_gated(x, gl, lam, z, h0, c=c)
    h, hl = orc.fwd(x, gl, lam, h0, c=c)
    assert _rel(y, h) < 1e-14 and np.array_equal(yl, hl)
    gated = orc.bwd_gated(dy, x, gl, lam, z, h0, dh_last, c=c)
    plain = orc.bwd(dy, x, gl, lam, h0, dh_last, c=c)
    for a, b in zip(gated[:4], plain):
        assert _rel(a, b) < 1e-13


def pin_gated_finite_differences(orc):
    rng = np.random.default_rng(25)
    B, L, D, c = 2, 5, 3, 0.8
    x, gl, lam = _rand_problem(rng, B, L, D, decay=(0.6, 0.97))
    z = 2.0 * rng.standard_normal((B, L, D))
    h0 = rng.standard_normal((B, D))
    dy = rng.standard_normal((B, L, D))
    dh_last = rng.standard_normal((B, D))
    dx, dgl, dlam, dh0, dz = orc.bwd_gated(dy, x, gl, lam, z, h0, dh_last, c=c)
    eps = 1e-6

    def loss(x_, gl_, lam_, z_, h0_):
        y, yl = orc.fwd_gated(x_, gl_, lam_, z_, h0_, c=c)
        return float(np.sum(dy * y) + np.sum(dh_last * yl))

    def fd(arr, which):
        out = np.empty_like(arr)
        args = [x, gl, lam, z, h0]
        for idx in np.ndindex(arr.shape):
            p = arr.copy(); p[idx] += eps
            m = arr.copy(); m[idx] -= eps
            ap, am = list(args), list(args)
            ap[which], am[which] = p, m
            out[idx] = (loss(*ap) - loss(*am)) / (2 * eps)
        return out

    for got, arr, which, name in ((dx, x, 0, "dx"), (dgl, gl, 1, "dgl"), (dlam, lam, 2, "dlambda"),
                                  (dz, z, 3, "dz"), (dh0, h0, 4, "dh0")):
        assert _rel(got, fd(arr, which)) < 1e-6, name


ALL_PINS = [
    pin_golden_forward,
    pin_geometric_closed_form,
    pin_alpha_zero,
    pin_alpha_one,
    pin_linearity,
    pin_bruteforce,
    pin_two_tree_scan,
    pin_left_padding,
    pin_split_resume,
    pin_bound,
    pin_golden_backward,
    pin_finite_differences,
    pin_gradient_linearity,
    pin_step,
    pin_steps,
    pin_varlen_is_zero_left_padding,
    pin_varlen_full_and_empty,
    pin_merge_limits,
    pin_merge_unit_gate,
    pin_gated_finite_differences,
]
