"""The oracle's pins catch plausible mistakes (CPU only).

Each case plants one mistake in a copy of the oracle's source (a transposed
operand, a dropped term, a wrong index or sign), loads the copy as a fresh
module, and runs the pins of ``test_oracle_pins`` against it: at least one pin
must fail.  The real oracle is never modified.
"""

import importlib.util
import os
import types

import pytest

import tests.test_oracle_pins as pins
from oracle import bcmt_oracle

SRC = open(bcmt_oracle.__file__).read()

MUTATIONS = {
    "W_O transposed": ("Hloc[b, t0:t1] = Hhat[b, t0:t1] @ w_o", "Hloc[b, t0:t1] = Hhat[b, t0:t1] @ w_o.T"),
    "Q projected with W_K": ("W_Q = np.ascontiguousarray(w_qkv[:, 0:D])", "W_Q = np.ascontiguousarray(w_qkv[:, D:2 * D])"),
    "no 1/sqrt(d_h)": ("/ math.sqrt(d_h) + mask", "+ mask"),
    "mask lets one future key in": ("np.full((Li, Li), -np.inf), k=1)", "np.full((Li, Li), -np.inf), k=2)"),
    "memory not shifted": ("C[b, i] = P[b, i - 1]", "C[b, i] = P[b, i]"),
    "decay exponent off by one": ("wgt = a ** (i - j)", "wgt = a ** (i - j + 1)"),
    "memory not normalised": ("M[b, i] = num / den", "M[b, i] = num"),
    "W_g transposed": ("G[b] = _sigmoid(Hloc[b] @ w_g)", "G[b] = _sigmoid(Hloc[b] @ w_g.T)"),
    "injection sign": ("Y[b, t0:t1] = Hloc[b, t0:t1] + G[b, t0:t1]", "Y[b, t0:t1] = Hloc[b, t0:t1] - G[b, t0:t1]"),
    "summary pools W_p-weighted tokens unnormalised": ("S[b, i] = Hb.T @ ab", "S[b, i] = Hb.T @ np.exp(sb)"),
    "bwd: softmax Jacobian term dropped": ("ds = ab * (g - np.dot(ab, g))", "ds = ab * g"),
    "bwd: reverse scan divides by Z_j": ("dS[j] += (a ** (i - j)) * dM[i] / Z[i]", "dS[j] += (a ** (i - j)) * dM[i] / Z[j]"),
    "bwd: shift not reversed": ("dP[i] = dC[i + 1]", "dP[i] = dC[i]"),
    "bwd: dK with untransposed scores": ("dK[b, t0:t1, cols] = dScore.T @ Qb", "dK[b, t0:t1, cols] = dScore @ Qb"),
    "bwd: decay gradient without the denominator term": ("d_decay += dM[i] * (dnum - M[b, i] * dden) / Z[i]", "d_decay += dM[i] * dnum / Z[i]"),
    "bwd: decay gradient exponent": ("w = (i - j) * a ** (i - j - 1)", "w = (i - j) * a ** (i - j)"),
    "bwd: gate derivative": ("dU[t0:t1] = dG * G[b, t0:t1] * (1.0 - G[b, t0:t1])", "dU[t0:t1] = dG * G[b, t0:t1]"),
}

PINS = [
    lambda: pins.test_worked_examples(0),
    lambda: pins.test_worked_examples(1),
    lambda: pins.test_single_block_is_dense_causal_attention(7, 7),
    lambda: pins.test_blockwise_attention_is_block_diagonal_sdpa(10, 4, 2),
    pins.test_pooling_weights_are_block_softmax,
    pins.test_decay_zero_memory_is_previous_summary,
    pins.test_denominator_closed_form,
    pins.test_memory_brute_force_token_sum,
    pins.test_causality,
    pins.test_block_never_sees_its_own_summary,
    pins.test_backward_finite_differences,
]


def _load_mutant(old, new):
    assert SRC.count(old) == 1, old
    mod = types.ModuleType("bcmt_oracle_mutant")
    mod.__file__ = "<mutant>"
    exec(compile(SRC.replace(old, new), "<mutant>", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTATIONS))
@pytest.mark.filterwarnings("ignore::RuntimeWarning")  # a mutant may divide by zero
def test_pins_catch_mutation(name, monkeypatch):
    mutant = _load_mutant(*MUTATIONS[name])
    monkeypatch.setattr(pins, "O", mutant)
    caught = []
    for pin in PINS:
        try:
            pin()
        except (AssertionError, FloatingPointError, ValueError, IndexError):
            caught.append(pin)
            break
    assert caught, f"no pin caught the planted mistake: {name}"
