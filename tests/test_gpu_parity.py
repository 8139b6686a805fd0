"""Parity of the CUDA path (through the C ABI) with the float64 oracle.

Bar (stated per test): per-row final objective within relative 1e-4 and
scales within relative 1e-4 on rows whose codes match, at least 99.9 % of
codes identical, and every difference starting at a near-tie of the
oracle's own values (``parity.lockstep``).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

from oracle import Options, group_target, objective, prepare_hessian, refine_layer  # noqa: E402
from synth import Layer, small_layer, tiny_layer  # noqa: E402
from tests.parity import compare_final, gpu_refine, lockstep  # noqa: E402

REL_F = 1e-4
REL_S = 1e-4
CODES_SAME = 0.999


@pytest.fixture(scope="module")
def jarq():
    from paper_2609_38599_gb300 import jarq as mod
    return mod


def oracle_run(lay, K, early_stop):
    prep = prepare_hessian(lay.H, lay.g)
    res = refine_layer(prep, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits,
                       Options(max_iters=K, early_stop=early_stop))
    return prep, res


@pytest.mark.parametrize("early_stop", [False, True])
def test_tiny_layer_parity(jarq, early_stop):
    """256x256, g=64, 3-bit, K=5: the tiny workload, whole layer."""
    lay = tiny_layer()
    prep, res = oracle_run(lay, 5, early_stop)
    S, Q, st = gpu_refine(lay, 5, early_stop=early_stop)
    assert st["status"] == 0
    m = compare_final(lay, prep, res, S, Q, st)
    assert m["codes_same"] >= CODES_SAME, m
    assert m["S_rel_max_same_rows"] <= REL_S, m
    assert m["F_rel_max_same_rows"] <= REL_F, m
    assert m["F_rel_all"] <= REL_F, m
    assert m["Lhost_rel"] <= 1e-5 and m["Lfinal_vs_oracle_state"] <= 1e-5, m
    assert m["gpu_no_worse_than_host"], m
    assert np.array_equal(st["iters"] > 0, np.ones(lay.dout, bool))
    if early_stop:
        agree = np.mean(st["iters"] == res.iters)
        assert agree >= 0.99, agree


@pytest.mark.parametrize("din,dout,g,bits,K", [
    (128, 100, 64, 3, 4),     # ragged rows (not a tile multiple)
    (256, 257, 128, 4, 3),    # two groups of 128, ragged rows
    (192, 70, 64, 2, 3),      # 2-bit, three groups, din not a multiple of 128
    (448, 33, 64, 3, 5),      # seven groups of 64
    (640, 129, 128, 3, 4),    # five groups of 128
    (1024, 300, 128, 4, 2),   # several K chunks per split
    (256, 96, 64, 6, 3),      # 6-bit: codes beyond 4 bits (wide integer dots)
    (384, 64, 128, 8, 2),     # 8-bit: codes need 16-bit staging
])
def test_shapes_parity(jarq, din, dout, g, bits, K):
    lay = small_layer(din, dout, g, bits, K=K, seed=din + dout + g)
    prep, res = oracle_run(lay, K, False)
    S, Q, st = gpu_refine(lay, K)
    m = compare_final(lay, prep, res, S, Q, st)
    assert m["codes_same"] >= CODES_SAME, m
    assert m["S_rel_max_same_rows"] <= REL_S and m["F_rel_max_same_rows"] <= REL_F, m
    assert m["F_rel_all"] <= REL_F, m
    assert m["gpu_no_worse_than_host"], m
    assert Q.min() >= 0 and Q.max() <= (1 << bits) - 1


def _many_group_layer(din, dout, g, bits, K, seed):
    """A layer with the small-layer recipe whose Hessian is accumulated on
    the GPU (torch generators), returned as NumPy arrays for the oracle."""
    from synth.layers import hessian_torch, rtn_host_torch, weights_torch
    H = hessian_torch(din, max(1, din // 16), 2, 20.0, 2 * din, 0.1, seed, "cuda")
    W = weights_torch(dout, din, 0.02, 0.005, 8.0, "normal", seed + 1, "cuda")
    S0, Q0, Z = rtn_host_torch(W, bits, g)
    n = lambda x: x.cpu().numpy()
    return Layer(f"many_{dout}x{din}_g{g}_w{bits}", n(W), n(H), n(S0), n(Q0), n(Z), bits, g, K)


@pytest.mark.parametrize("din,dout,g,bits,K", [
    (2304, 40, 64, 3, 2),     # 36 groups: the scale solve with G > 32
    (4224, 24, 128, 4, 2),    # 33 groups of 128
    (8192, 12, 64, 3, 1),     # 128 groups: the largest G the solve accepts
])
def test_many_groups_parity(jarq, din, dout, g, bits, K):
    lay = _many_group_layer(din, dout, g, bits, K, seed=din + g)
    prep, res = oracle_run(lay, K, False)
    S, Q, st = gpu_refine(lay, K)
    assert st["status"] == 0
    m = compare_final(lay, prep, res, S, Q, st)
    assert m["codes_same"] >= CODES_SAME, m
    assert m["S_rel_max_same_rows"] <= REL_S and m["F_rel_max_same_rows"] <= REL_F, m
    assert m["F_rel_all"] <= REL_F, m
    assert m["gpu_no_worse_than_host"], m


@pytest.mark.parametrize("early_stop", [False, True])
def test_two_chain_sweep_parity(jarq, early_stop):
    """10200 rows, din 256, g = 128: one phase product needs 80 x 2 = 160 CTAs,
    more than one wave, so the sweep runs as two chains over the row halves
    (5120 and 5080 rows, the second ending in a ragged tile).  Every row is
    compared; with the early stop on, also the stopping iterations."""
    K = 4 if early_stop else 2
    lay = small_layer(256, 10200, 128, 3, K=K, seed=77)
    prep, res = oracle_run(lay, K, early_stop)
    S, Q, st = gpu_refine(lay, K, early_stop=early_stop)
    if early_stop:
        assert np.mean(st["iters"] == res.iters) >= 0.99
    assert st["status"] == 0
    m = compare_final(lay, prep, res, S, Q, st)
    assert m["codes_same"] >= CODES_SAME, m
    assert m["S_rel_max_same_rows"] <= REL_S and m["F_rel_max_same_rows"] <= REL_F, m
    assert m["F_rel_all"] <= REL_F, m
    assert m["gpu_no_worse_than_host"], m


def test_lockstep_tiny_every_difference_is_a_near_tie(jarq):
    lay = tiny_layer()

    def step(S, Q):
        S2, Q2, _ = gpu_refine(lay, 1, S=S, Q=Q)
        return S2, Q2

    recs = lockstep(lay, 5, step)
    assert len(recs) == 5


def test_objective_entry_point(jarq):
    lay = small_layer(384, 77, 128, 3, seed=21)
    prep = prepare_hessian(lay.H, lay.g)
    F_or = objective(prep, lay.W, lay.S0, lay.Q0, lay.Z)
    dev = "cuda"
    hess = jarq.prepare(torch.as_tensor(lay.H, device=dev), lay.g)
    F = jarq.objective(hess, torch.as_tensor(lay.W, device=dev), torch.as_tensor(lay.S0, device=dev),
                       torch.as_tensor(lay.Q0, device=dev), torch.as_tensor(lay.Z, device=dev),
                       lay.bits).cpu().numpy()
    np.testing.assert_allclose(F, F_or, rtol=1e-5)
    # host buffers give the same numbers
    F2 = jarq.objective(hess, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits)
    np.testing.assert_allclose(F2, F, rtol=0, atol=0)
    hess.close()


@pytest.mark.parametrize("din,dout,g,bits", [(384, 77, 128, 3), (320, 130, 64, 4)])
def test_residual_product_elementwise(jarq, din, dout, g, bits):
    """The split-precision tensor-core product H r (Eq. conditional_residual's
    (H r)_i for every group) against the oracle's float64 group slices, element
    by element.  The kernel's residual is float32 and its bf16 x 3 products
    drop terms below 2^-24, so the error is bounded relative to |H| |r|."""
    lay = small_layer(din, dout, g, bits, seed=31)
    prep = prepare_hessian(lay.H, lay.g)
    C = lay.Q0.astype(np.float64) - np.repeat(lay.Z, g, axis=1)
    r = lay.W.astype(np.float64) - np.repeat(lay.S0.astype(np.float64), g, axis=1) * C
    ref = np.concatenate([group_target(prep, r, lay.S0[:, i], C[:, i * g:(i + 1) * g], i)[0]
                          for i in range(din // g)], axis=1)
    scale = np.abs(r) @ np.abs(prep.H)
    dev = "cuda"
    hess = jarq.prepare(torch.as_tensor(lay.H, device=dev), lay.g)
    HR = jarq.residual_product(hess, torch.as_tensor(lay.W, device=dev),
                               torch.as_tensor(lay.S0, device=dev), torch.as_tensor(lay.Q0, device=dev),
                               torch.as_tensor(lay.Z, device=dev), lay.bits).cpu().numpy()
    hess.close()
    assert HR.shape == (dout, din)
    assert np.all(np.abs(HR - ref) <= 4e-6 * scale + 1e-30)


def test_host_buffers_match_device_buffers(jarq):
    lay = small_layer(256, 96, 64, 3, seed=22)
    Sd, Qd, std = gpu_refine(lay, 3)
    Sh, Qh, sth = gpu_refine(lay, 3, host=True)
    assert np.array_equal(Qd, Qh)
    assert np.array_equal(Sd, Sh)
    np.testing.assert_array_equal(std["L_final"], sth.L_final)


def test_k0_returns_host_state(jarq):
    lay = small_layer(128, 40, 64, 3, seed=23)
    S, Q, st = gpu_refine(lay, 0)
    assert np.array_equal(Q, lay.Q0) and np.array_equal(S, lay.S0)
    np.testing.assert_allclose(st["L_final"], st["L_host"], rtol=0)


def test_empty_layer_is_a_no_op(jarq):
    """dout = 0 (no output rows): every layer entry point returns JARQ_OK and
    touches nothing; the pointers may then be NULL."""
    import ctypes
    lay = tiny_layer()
    hess = jarq.prepare(torch.as_tensor(lay.H, device="cuda"), lay.g)
    lib = jarq.library()
    h = hess.handle
    o = jarq.default_options(max_iters=3)
    OK = 0
    assert lib.jarq_refine_layer(h, None, None, None, None, 0, lay.bits, ctypes.byref(o), None, None) == OK
    assert lib.jarq_objective(h, None, None, None, None, 0, lay.bits, None, None) == OK
    assert lib.jarq_objective_noalloc(h, None, None, None, None, 0, lay.bits, None, None) == OK
    assert lib.jarq_residual_product(h, None, None, None, None, 0, lay.bits, None, None) == OK
    assert lib.jarq_fit_scales(h, None, None, None, None, 0, lay.bits, 0, 3, None, None, None) == OK
    assert lib.jarq_multicode_probe(h, None, None, None, None, 0, lay.bits, 0,
                                    None, None, None, None, None, None) == OK
    # the mu-target still needs its two Gram matrices (not read when dout = 0)
    Hd = torch.as_tensor(lay.H, device="cuda")
    assert lib.jarq_refine_layer_mu(h, None, None, None, None, 0, lay.bits, Hd.data_ptr(),
                                    Hd.data_ptr(), 0.5, 0.0, ctypes.byref(o), None, None) == OK
    assert lib.jarq_refine_layer_mu(h, None, None, None, None, 0, lay.bits, None, None, 0.5, 0.0,
                                    ctypes.byref(o), None, None) == jarq.JARQ_ERR_ARG
    # real buffers with dout = 0 stay untouched
    S = torch.as_tensor(lay.S0[:1], device="cuda").clone()
    Q = torch.as_tensor(lay.Q0[:1], device="cuda").clone()
    W = torch.as_tensor(lay.W[:1], device="cuda")
    Z = torch.as_tensor(lay.Z[:1], device="cuda")
    assert lib.jarq_refine_layer(h, W.data_ptr(), S.data_ptr(), Q.data_ptr(), Z.data_ptr(), 0,
                                 lay.bits, ctypes.byref(o), None, None) == OK
    torch.cuda.synchronize()
    assert np.array_equal(S.cpu().numpy(), lay.S0[:1]) and np.array_equal(Q.cpu().numpy(), lay.Q0[:1])
    hess.close()


def test_format_preserved(jarq):
    lay = small_layer(256, 64, 64, 4, seed=24)
    Z0 = lay.Z.copy()
    dev = "cuda"
    hess = jarq.prepare(torch.as_tensor(lay.H, device=dev), lay.g)
    Z = torch.as_tensor(lay.Z, device=dev)
    S = torch.as_tensor(lay.S0, device=dev).clone()
    Q = torch.as_tensor(lay.Q0, device=dev).clone()
    jarq.refine(hess, torch.as_tensor(lay.W, device=dev), S, Q, Z, lay.bits, max_iters=3)
    assert np.array_equal(Z.cpu().numpy(), Z0)
    assert int(Q.max()) <= 15 and int(Q.min()) >= 0
    assert tuple(S.shape) == lay.S0.shape
    hess.close()


def test_bad_codes_rejected_before_any_update(jarq):
    lay = small_layer(128, 16, 64, 3, seed=25)
    Q = lay.Q0.copy()
    Q[3, 5] = 9          # outside [0, 7]
    S = lay.S0.copy()
    from paper_2609_38599_gb300 import jarq as J
    hess = J.prepare(lay.H, lay.g)
    st = J.refine(hess, lay.W, S, Q, lay.Z, 3, max_iters=2, raise_on_error=False)
    assert st.status == J.JARQ_ERR_ARG
    assert np.array_equal(S, lay.S0) and Q[3, 5] == 9
    Zb = lay.Z.copy()
    Zb[0, 0] = -1
    st = J.refine(hess, lay.W, lay.S0.copy(), lay.Q0.copy(), Zb, 3, max_iters=2,
                  raise_on_error=False)
    assert st.status == J.JARQ_ERR_ARG
    hess.close()


def test_not_spd_hessian_reported(jarq):
    H = np.eye(64, dtype=np.float32)
    H[40, 40] = -1.0
    from paper_2609_38599_gb300 import jarq as J
    with pytest.raises(J.JarqError) as ei:
        J.prepare(H, 64)
    assert ei.value.status == J.JARQ_ERR_NOT_SPD


def test_zero_group_takes_ridge_and_nan_row_is_numerical(jarq):
    lay = small_layer(256, 8, 64, 3, seed=26)
    Q = lay.Q0.copy()
    Q[2, 64:128] = lay.Z[2, 1]          # c_i = 0: singular Gram -> ridge
    W = lay.W.copy()
    W[5, 7] = np.nan                    # nonfinite target -> numerical error
    lay2 = Layer(lay.name, W, lay.H, lay.S0, Q, lay.Z, 3, 64, 2)
    S, Qg, st = gpu_refine(lay2, 2)
    assert st["status"] == 3            # JARQ_ERR_NUMERICAL for the call
    assert st["row_status"][5] == 3 and np.all(np.delete(st["row_status"], 5) == 0)
    assert st["ridge_hits"][2] >= 1
    assert np.array_equal(S[5], lay.S0[5]) and np.array_equal(Qg[5], Q[5])
    # the other rows still match the oracle
    prep = prepare_hessian(lay.H, lay.g)
    rows = np.array([0, 1, 3, 4, 6, 7])
    res = refine_layer(prep, W[rows], lay.S0[rows], Q[rows], lay.Z[rows], 3,
                       Options(max_iters=2, early_stop=False))
    assert np.mean(Qg[rows] == res.Q) >= CODES_SAME


def test_small_scale_group_keeps_codes(jarq):
    lay = small_layer(256, 12, 64, 3, seed=27)
    # zero a group's codes-minus-zero so its refit scale is 0 (below eps)
    Q = lay.Q0.copy()
    Q[:, 64:128] = lay.Z[:, 1:2]
    lay2 = Layer(lay.name, lay.W, lay.H, lay.S0, Q, lay.Z, 3, 64, 1)
    S, Qg, st = gpu_refine(lay2, 1)
    assert np.all(np.abs(S[:, 1]) <= 1e-6)
    assert np.array_equal(Qg[:, 64:128], Q[:, 64:128])


def test_bounded_wait_reports_timeout_and_context_survives(jarq):
    """A device wait that nothing completes gives up after its poll limit and
    the call reports JARQ_ERR_TIMEOUT, through the status word and mapping
    every kernel's bounded waits use; the context stays usable afterwards:
    the tiny layer still refines as the oracle does."""
    assert jarq.selftest_wait_timeout() == jarq.JARQ_ERR_TIMEOUT
    lay = tiny_layer()
    prep, res = oracle_run(lay, 2, False)
    S, Q, st = gpu_refine(lay, 2, early_stop=False)
    assert st["status"] == 0
    m = compare_final(lay, prep, res, S, Q, st)
    assert m["codes_same"] >= CODES_SAME, m
    assert m["F_rel_all"] <= REL_F, m
