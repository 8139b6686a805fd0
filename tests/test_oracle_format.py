"""Pins of the write-back formats and of the ridge-acceptance variant.

App. E "Early stopping" (the returned weights are cast to the model's
dtype), Sec. 3.1 (b-bit codes), App. E "Representing Negative Scales" and
App. G Remark ridge-acceptance.  Each pin checks the oracle against
something other than itself: literal bit patterns, an integer big-number
construction, float16 conversion by numpy, bfloat16 by float32 bit
manipulation, and the objective itself.
"""
import numpy as np
import pytest

from oracle import (Options, canonicalize, dequantize, dequantize_cast, objective, pack_codes,
                    prepare_hessian, refine_layer, round_to_bfloat16, scale_system, unpack_codes)
from synth import small_layer


def test_pack_codes_literal_words():
    """Nibbles and bytes land little-endian in 32-bit words; 3-bit codes
    straddle word boundaries."""
    q4 = np.array([[1, 2, 3, 4, 5, 6, 7, 8]], dtype=np.uint8)
    assert pack_codes(q4, 4).tolist() == [[0x87654321]]
    q8 = np.array([[0x11, 0x22, 0x33, 0x44, 0x55]], dtype=np.uint8)
    assert pack_codes(q8, 8).tolist() == [[0x44332211, 0x00000055]]
    q3 = np.full((1, 11), 7, dtype=np.uint8)          # 33 one bits
    assert pack_codes(q3, 3).tolist() == [[0xFFFFFFFF, 0x00000001]]
    q3b = np.array([[0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 5]], dtype=np.uint8)   # bits 30..32 = 101
    assert pack_codes(q3b, 3).tolist() == [[0x40000000, 0x00000001]]


@pytest.mark.parametrize("bits", [2, 3, 4, 5, 7, 8])
def test_pack_codes_matches_big_integer_stream(bits):
    rng = np.random.default_rng(bits)
    Q = rng.integers(0, 1 << bits, size=(5, 77), dtype=np.uint8)
    P = pack_codes(Q, bits)
    for j in range(Q.shape[0]):
        stream = sum(int(Q[j, k]) << (k * bits) for k in range(Q.shape[1]))
        words = [(stream >> (32 * w)) & 0xFFFFFFFF for w in range(P.shape[1])]
        assert P[j].tolist() == words
    assert np.array_equal(unpack_codes(P, Q.shape[1], bits), Q)


def test_bfloat16_rounding_ties_to_even_and_matches_float32_bit_rounding():
    assert round_to_bfloat16(1 + 2.0 ** -8) == 1.0                 # tie, even below
    assert round_to_bfloat16(1 + 3 * 2.0 ** -8) == 1 + 2.0 ** -6   # tie, even above
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(10000) * 0.03).astype(np.float32)
    b = x.view(np.uint32).astype(np.uint64)
    r = ((b + 0x7FFF + ((b >> 16) & 1)) >> 16) << 16               # round-to-nearest-even on the bits
    ref = r.astype(np.uint32).view(np.float32).astype(np.float64)
    assert np.array_equal(round_to_bfloat16(x.astype(np.float64)), ref)


def test_dequantize_cast_is_one_rounding_of_the_exact_weights():
    lay = small_layer(64, 6, 16, 3, seed=3)
    S = -lay.S0.astype(np.float32) * 1.37                          # signed, arbitrary float32 scales
    exact = dequantize(S, lay.Q0, lay.Z, 16)
    assert np.array_equal(dequantize_cast(S, lay.Q0, lay.Z, 16, "float16"), exact.astype(np.float16))
    assert np.array_equal(dequantize_cast(S, lay.Q0, lay.Z, 16, "float32"), exact.astype(np.float32))
    # canonicalisation changes no weight (Eq. canonicalization_equivalence)
    S2, Q2, Z2 = canonicalize(S, lay.Q0, lay.Z, 3)
    assert np.all(S2 >= 0) and Q2.max() <= 7 and Z2.max() <= 7
    assert np.array_equal(dequantize(S2, Q2, Z2, 16), exact)


def _ridge_layer():
    """A row whose starting scales are the exact least-squares scales of its
    codes, with one group at its zero point (singular Gram matrix, so the
    ridge fires) and H scaled so that the ridge bias is visible."""
    lay = small_layer(64, 4, 16, 3, seed=5, rank=4, tokens=400)
    H = lay.H.astype(np.float64) * 1e-4
    Q = lay.Q0.copy()
    Q[1, 16:32] = lay.Z[1, 1]
    prep = prepare_hessian(H, 16)
    Gram, rhs = scale_system(prep, lay.W[1:2], Q[1:2], lay.Z[1:2])
    keep = [0, 2, 3]
    s = lay.S0[1].astype(np.float64).copy()
    s[keep] = np.linalg.solve(Gram[0][np.ix_(keep, keep)], rhs[0][keep])
    S0 = lay.S0.astype(np.float64).copy()
    S0[1] = s
    return lay, prep, S0, Q


def test_ridge_acceptance_keeps_previous_scales_when_the_ridge_would_raise_F():
    """Remark ridge-acceptance: without it, the ridge solve can raise F_j at
    a scale update; with it, the previous scales are kept and F_j does not
    rise."""
    lay, prep, S0, Q = _ridge_layer()
    F0 = objective(prep, lay.W, S0, Q, lay.Z)
    for accept in (False, True):
        trace = []
        res = refine_layer(prep, lay.W, S0, Q, lay.Z, 3,
                           Options(max_iters=1, early_stop=False, fp32_scales=False,
                                   ridge_accept=accept), trace=trace)
        sc = trace[0]
        assert res.ridge_hits[1] == 1
        L1 = sc["L"][list(sc["rows"]).index(1)]
        if accept:
            assert L1 <= F0[1]
            assert np.array_equal(sc["S"][list(sc["rows"]).index(1)], S0[1])
        else:
            assert L1 > F0[1] * (1 + 1e-9)
