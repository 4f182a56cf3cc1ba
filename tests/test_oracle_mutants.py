"""CPU: the oracle pins are strong enough to catch plausible mistakes.

Each case plants one mistake in a temporary copy of the oracle's C source (a
dropped term, a wrong sign, a transposed operand, an ignored input), builds it
and checks that at least one pin of ``oracle_pins.ALL_PINS`` fails on it. The
real oracle is never modified."""
import os

import pytest

import oracle
from oracle_pins import ALL_PINS

# (name, exact text in blr_oracle.c, replacement, occurrences to replace or -1 for all)
MUTANTS = [
    ("recurrence gate sign", "g.r = sigmoid(rho);", "g.r = sigmoid(-rho);", 1),
    ("input gate dropped", "sqrt(1.0 - g.alpha * g.alpha) * g.i;", "sqrt(1.0 - g.alpha * g.alpha);", 1),
    ("decay constant c dropped", "g.alpha = exp(-c * s * g.r);", "g.alpha = exp(-s * g.r);", 1),
    ("alpha for alpha^2 in beta", "sqrt(1.0 - g.alpha * g.alpha) * g.i", "sqrt(1.0 - g.alpha) * g.i", 1),
    ("softplus as plain exp", "return log1p(exp(z));", "return exp(z);", 1),
    ("operands of the recurrence swapped", "state = g.alpha * state + g.beta * x[row * D + d];",
     "state = g.beta * state + g.alpha * x[row * D + d];", 1),
    ("h0 ignored in forward", "double state = h0 ? h0[b * D + d] : 0.0;", "double state = 0.0;", 1),
    ("reverse carry without alpha", "g_next = gt.alpha * g;", "g_next = g;", 1),
    ("sign of the normalisation term", "hprev - gt.alpha * gt.i * xt / norm", "hprev + gt.alpha * gt.i * xt / norm", 1),
    ("sigmoid derivative dropped (rho)", "dL_dr * gt.r * (1.0 - gt.r)", "dL_dr * gt.r", 1),
    ("sigmoid derivative dropped (iota)", "dL_di * gt.i * (1.0 - gt.i)", "dL_di", 1),
    ("softplus derivative dropped", "* ds_dlambda;", ";", 1),
    ("dh_last ignored", "double g_next = dh_last ? dh_last[b * D + d] : 0.0;", "double g_next = 0.0;", 1),
    ("rho and iota columns transposed", "gl[row * 2 * D + d], gl[row * 2 * D + D + d]",
     "gl[row * 2 * D + D + d], gl[row * 2 * D + d]", -1),
    ("h_{t-1} read one step late", "dx[row * D + d] = state; /* h_{t-1} */\n        gates_t gt = step_gates(c, s, gl[row * 2 * D + d], gl[row * 2 * D + D + d]);\n        state = gt.alpha * state + gt.beta * x[row * D + d];",
     "gates_t gt = step_gates(c, s, gl[row * 2 * D + d], gl[row * 2 * D + D + d]);\n        state = gt.alpha * state + gt.beta * x[row * D + d];\n        dx[row * D + d] = state;", 1),
    ("merge gate without its z factor", "y[k] = h[k] * (z[k] * sigmoid(z[k]));", "y[k] = h[k] * sigmoid(z[k]);", 1),
    ("merge slope without the z (1 - sigmoid) term", "(sg * (1.0 + z[k] * (1.0 - sg)))", "(sg * (1.0 + (1.0 - sg)))", 1),
    ("merge passes dy through ungated", "dh[k] = dy[k] * (z[k] * sg);", "dh[k] = dy[k];", 1),
]


@pytest.mark.parametrize("name,old,new,count", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_planted_mistake(tmp_path, name, old, new, count):
    with open(oracle.SOURCE) as f:
        src = f.read()
    assert src.count(old) >= 1, f"mutation anchor not found: {old!r}"
    mutated = src.replace(old, new) if count < 0 else src.replace(old, new, count)
    path = tmp_path / "mutant.c"
    path.write_text(mutated)
    lib = oracle.build(str(path), str(tmp_path / "libmutant.so"), openmp=False)
    orc = oracle.Oracle(lib)
    caught = []
    for pin in ALL_PINS:
        try:
            pin(orc)
        except (AssertionError, FloatingPointError, ValueError):
            caught.append(pin.__name__)
    assert caught, f"no pin caught the planted mistake: {name}"
