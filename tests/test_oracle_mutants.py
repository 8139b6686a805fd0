"""Planted mistakes in the oracle must be caught by its pins.

Each case patches one plausible error into ``oracle.jarq_oracle`` (a
transposed factor, a dropped term, a wrong sign,
a skipped zero point, a missing cross term) and re-runs pins from
``test_oracle_pins``; at least one must fail.  Everything here runs on the
CPU.
"""
import numpy as np
import pytest

import oracle.jarq_oracle as jo
import tests.test_oracle_pins as pins

PIN_SET = [
    pins.test_multicode_babai_step_and_refit,
    pins.test_staleness_refit_unlocks_descent,
    pins.test_staleness_host_grid_optimum,
    pins.test_multicode_single_code_neighbours,
    pins.test_h_form_matches_paper_literal_qr_form,
    pins.test_accepted_proposals_strictly_decrease,
    pins.test_monotone_descent_every_half_step,
    pins.test_single_group_scale_is_scalar_least_squares,
]


def _transposed_babai(R_i, v, z, qmax):
    rows, g = v.shape
    q = np.zeros((rows, g))
    x = np.zeros((rows, g))
    for l in range(g - 1, -1, -1):
        acc = v[:, l] - (q[:, l + 1:] - z[:, None]) @ R_i[l + 1:, l]
        x[:, l] = acc / R_i[l, l]
        q[:, l] = np.clip(np.rint(z + x[:, l]), 0, qmax)
    return q, x


def _babai_without_zero_point(R_i, v, z, qmax):
    rows, g = v.shape
    q = np.zeros((rows, g))
    x = np.zeros((rows, g))
    for l in range(g - 1, -1, -1):
        acc = v[:, l] - q[:, l + 1:] @ R_i[l, l + 1:]
        x[:, l] = acc / R_i[l, l]
        q[:, l] = np.clip(np.rint(z + x[:, l]), 0, qmax)
    return q, x


def _target_without_own_group(prep, r, S_i, C_i, i):
    g = prep.g
    si = slice(i * g, (i + 1) * g)
    Hr_i = r @ prep.H[:, si]
    return Hr_i, Hr_i


def _target_wrong_sign(prep, r, S_i, C_i, i):
    g = prep.g
    si = slice(i * g, (i + 1) * g)
    Hr_i = r @ prep.H[:, si]
    return Hr_i, Hr_i - (S_i[:, None] * C_i) @ prep.H[si, si]


def _rhs_without_H(prep, W, Q, Z):
    Gram, _ = ORIG_SCALE_SYSTEM(prep, W, Q, Z)
    g = prep.g
    C = np.asarray(Q, dtype=np.float64) - np.repeat(np.asarray(Z, dtype=np.float64), g, axis=1)
    rhs = (C * np.asarray(W, dtype=np.float64)).reshape(C.shape[0], -1, g).sum(-1)
    return Gram, rhs


def _gram_diagonal_only(prep, W, Q, Z):
    Gram, rhs = ORIG_SCALE_SYSTEM(prep, W, Q, Z)
    return Gram * np.eye(Gram.shape[1])[None], rhs


ORIG_SCALE_SYSTEM = jo.scale_system


MUTANTS = {
    "babai_uses_transposed_R": ("babai_proposal", _transposed_babai),
    "babai_drops_zero_point": ("babai_proposal", _babai_without_zero_point),
    "target_drops_own_group_term": ("group_target", _target_without_own_group),
    "target_wrong_sign": ("group_target", _target_wrong_sign),
    "rhs_without_H": ("scale_system", _rhs_without_H),
    "gram_drops_cross_terms": ("scale_system", _gram_diagonal_only),
}


def _run_pins(golden_dir):
    failures = 0
    for pin in PIN_SET:
        try:
            if "golden_dir" in pin.__code__.co_varnames[:pin.__code__.co_argcount]:
                pin(golden_dir)
            else:
                pin()
        except (AssertionError, ValueError, np.linalg.LinAlgError, IndexError):
            failures += 1
    return failures


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name, golden_dir, monkeypatch):
    attr, fn = MUTANTS[name]
    monkeypatch.setattr(jo, attr, fn)
    if hasattr(pins, attr):
        monkeypatch.setattr(pins, attr, fn)
    assert _run_pins(golden_dir) >= 1, f"no pin caught mutant {name}"


def test_unmutated_oracle_passes_pin_set(golden_dir):
    assert _run_pins(golden_dir) == 0
