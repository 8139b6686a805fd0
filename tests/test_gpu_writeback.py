"""Write-back post-passes and the ridge-acceptance variant on the GPU,
against the oracle (bit-exact for the integer and rounding work).

App. E "Representing Negative Scales" (Eq. canonicalization), App. E "Early
stopping" (the refined weights cast to the model's dtype), Sec. 3.1 (b-bit
codes), App. G Remark ridge-acceptance.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

from oracle import (Options, canonicalize, dequantize_cast, pack_codes, prepare_hessian,  # noqa: E402
                    refine_layer, scale_system)
from synth import small_layer  # noqa: E402


@pytest.fixture(scope="module")
def jarq():
    from paper_2609_38599_gb300 import jarq as J
    return J


def _signed_state(dout, din, g, bits, seed):
    rng = np.random.default_rng(seed)
    G = din // g
    S = (rng.standard_normal((dout, G)) * 0.01).astype(np.float32)   # about half negative
    Q = rng.integers(0, 1 << bits, size=(dout, din), dtype=np.uint8)
    Z = rng.integers(0, 1 << bits, size=(dout, G)).astype(np.int32)
    return S, Q, Z


@pytest.mark.parametrize("dout,din,g,bits", [(130, 384, 128, 3), (77, 192, 64, 4), (5, 96, 32, 8)])
def test_canonicalize_bit_exact(jarq, dout, din, g, bits):
    S, Q, Z = _signed_state(dout, din, g, bits, seed=dout)
    S2, Q2, Z2 = canonicalize(S.astype(np.float64), Q, Z, bits)
    t = lambda a: torch.as_tensor(a).cuda()
    Sd, Qd, Zd = t(S), t(Q), t(Z)
    jarq.canonicalize(Sd, Qd, Zd, g, bits)
    assert np.array_equal(Sd.cpu().numpy(), S2.astype(np.float32))
    assert np.array_equal(Qd.cpu().numpy(), Q2)
    assert np.array_equal(Zd.cpu().numpy(), Z2)
    assert (S2 >= 0).all()


@pytest.mark.parametrize("dtype", ["float32", "float16", "bfloat16"])
def test_dequantize_bit_exact(jarq, dtype):
    S, Q, Z = _signed_state(96, 256, 64, 4, seed=9)
    ref = dequantize_cast(S, Q, Z, 64, dtype)
    t = lambda a: torch.as_tensor(a).cuda()
    out = jarq.dequantize(t(S), t(Q), t(Z), 64, 4, dtype).float().cpu().numpy().astype(np.float64)
    assert np.array_equal(out, np.asarray(ref, dtype=np.float64))


@pytest.mark.parametrize("bits", [2, 3, 4, 5, 6, 7, 8])
def test_pack_codes_bit_exact(jarq, bits):
    rng = np.random.default_rng(bits)
    Q = rng.integers(0, 1 << bits, size=(33, 203), dtype=np.uint8)    # ragged: 203 b not a multiple of 32
    ref = pack_codes(Q, bits)
    got = jarq.pack_codes(torch.as_tensor(Q).cuda(), bits).cpu().numpy().view(np.uint32)
    assert np.array_equal(got, ref)


def test_writeback_rejects_bad_input(jarq):
    S, Q, Z = _signed_state(8, 128, 64, 3, seed=1)
    lib = jarq.library()
    # host pointers
    assert lib.jarq_pack_codes(Q.ctypes.data, 8, 128, 3, Q.ctypes.data, None) == jarq.JARQ_ERR_ARG
    # a code outside [0, qmax] is rejected before any change
    Qd = torch.as_tensor(Q).cuda()
    Qd[3, 5] = 8
    Sd, Zd = torch.as_tensor(S).cuda(), torch.as_tensor(Z).cuda()
    S0 = Sd.clone()
    with pytest.raises(jarq.JarqError):
        jarq.canonicalize(Sd, Qd, Zd, 64, 3)
    assert torch.equal(Sd, S0)


def test_ridge_acceptance_matches_oracle(jarq):
    """A row whose starting scales are its exact least-squares scales and
    whose Gram matrix is singular (one group at its zero point, H scaled so
    the ridge bias shows): the ridge solve raises F, so with the option the
    previous scales are kept, without it they are not (App. G Remark
    ridge-acceptance); codes and scales match the oracle either way."""
    lay = small_layer(256, 4, 64, 3, seed=5, rank=8, tokens=1200)
    H = (lay.H.astype(np.float64) * 1e-4).astype(np.float32)
    Q = lay.Q0.copy()
    Q[1, 64:128] = lay.Z[1, 1]
    prep = prepare_hessian(H, 64)
    Gram, rhs = scale_system(prep, lay.W[1:2], Q[1:2], lay.Z[1:2])
    keep = [0, 2, 3]
    S0 = lay.S0.astype(np.float32).copy()
    S0[1, keep] = np.linalg.solve(Gram[0][np.ix_(keep, keep)], rhs[0][keep]).astype(np.float32)
    for accept in (0, 1):
        res = refine_layer(prep, lay.W, S0, Q, lay.Z, 3,
                           Options(max_iters=1, early_stop=False, ridge_accept=bool(accept)))
        t = lambda a: torch.as_tensor(np.ascontiguousarray(a)).cuda()
        hess = jarq.prepare(t(H), 64)
        S, Qd = t(S0), t(Q)
        st = jarq.refine(hess, t(lay.W), S, Qd, t(lay.Z), 3, max_iters=1, early_stop=0,
                         ridge_accept=accept, raise_on_error=False)
        hess.close()
        Sg = S.cpu().numpy()
        assert int(st.ridge_hits.cpu()[1]) == 1
        assert np.array_equal(Qd.cpu().numpy(), res.Q)
        np.testing.assert_allclose(Sg, res.S, rtol=1e-6)
        if accept:
            assert np.array_equal(Sg[1], S0[1])
        else:
            assert not np.array_equal(Sg[1], S0[1])
