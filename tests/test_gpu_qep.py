"""Refinement on the propagation-corrected (mu) target through the C ABI
against the oracle (App. "Propagation-Corrected Targets and QEP").

Both sides read the same float32 H (= X~^T X~ / n + nu2 I), K (= X~^T X / n)
and XX (= X^T X / n).  The oracle forms W_corr = W + (1 - mu) H^{-1}
X~^T (X - X~) W (Eq. w-corr) by a dense float64 solve and refines it with the
constant c_j in its objective; the CUDA path never inverts H: it projects by
K and XX on the tensor cores and combines.  Same bar as the main target:
>= 99.9 % of codes identical, scales and objectives within relative 1e-4 on
rows whose codes match, reported objectives within 1e-5 of the oracle's
objective of the same state.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

from oracle import Options, objective, prepare_hessian, refine_mu  # noqa: E402
from synth.qep import mu_layer  # noqa: E402


@pytest.fixture(scope="module")
def jarq():
    from paper_2609_38599_gb300 import jarq as mod
    return mod


def mu_compare(lay, mu, res, Wc, c, S_gpu, Q_gpu, st):
    prep = prepare_hessian(lay.H, lay.g)
    same_rows = np.all(Q_gpu == res.Q, axis=1)
    rel_S = np.abs(S_gpu - res.S) / np.maximum(np.abs(res.S), 1e-30)
    F_gpu_state = objective(prep, Wc, S_gpu, Q_gpu, lay.Z) + c
    return dict(
        codes_same=float(np.mean(Q_gpu == res.Q)),
        rows_same=float(np.mean(same_rows)),
        S_rel_max_same_rows=float(rel_S[same_rows].max()) if same_rows.any() else 0.0,
        F_rel_max_same_rows=float(np.max(np.abs(F_gpu_state[same_rows] - res.L_final[same_rows])
                                         / np.abs(res.L_final[same_rows]))) if same_rows.any() else 0.0,
        Lfinal_vs_oracle_state=float(np.max(np.abs(st.L_final - F_gpu_state) / np.abs(F_gpu_state))),
        Lhost_rel=float(np.max(np.abs(st.L_host - res.L_host) / np.abs(res.L_host))),
        gpu_no_worse_than_host=bool(np.all(F_gpu_state <= res.L_host * (1 + 1e-5))),
    )


def run_both(jarq, lay, mu, K_iters, early_stop):
    res, Wc, c = refine_mu(lay.H, lay.K, lay.XX, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits, lay.g, mu,
                           lay.nu2, Options(max_iters=K_iters, early_stop=early_stop))
    dev = "cuda"
    hess = jarq.prepare(torch.as_tensor(lay.H, device=dev), lay.g)
    S = torch.as_tensor(lay.S0, device=dev).clone()
    Q = torch.as_tensor(lay.Q0, device=dev).clone()
    st = jarq.refine_mu(hess, torch.as_tensor(lay.W, device=dev), S, Q,
                        torch.as_tensor(lay.Z, device=dev), lay.bits,
                        torch.as_tensor(lay.K, device=dev), torch.as_tensor(lay.XX, device=dev),
                        mu, lay.nu2, max_iters=K_iters, early_stop=int(early_stop))
    torch.cuda.synchronize()
    hess.close()

    class St:
        pass
    s = St()
    s.L_host, s.L_final = st.L_host.cpu().numpy(), st.L_final.cpu().numpy()
    s.iters = st.iters.cpu().numpy()
    return res, Wc, c, S.cpu().numpy(), Q.cpu().numpy(), s


@pytest.mark.parametrize("din,dout,g,bits,mu,K_iters,early_stop", [
    (256, 96, 64, 3, 0.5, 4, False),
    (384, 130, 128, 4, 0.0, 3, False),
    (256, 77, 64, 3, 0.8, 5, True),
    (512, 64, 128, 3, 0.25, 3, True),
])
def test_mu_target_parity(jarq, din, dout, g, bits, mu, K_iters, early_stop):
    lay = mu_layer(din, dout, g, bits, K_iters=K_iters, drift=0.08, seed=din + dout)
    res, Wc, c, S, Q, st = run_both(jarq, lay, mu, K_iters, early_stop)
    m = mu_compare(lay, mu, res, Wc, c, S, Q, st)
    print(m)
    assert m["codes_same"] >= 0.999, m
    assert m["S_rel_max_same_rows"] <= 1e-4 and m["F_rel_max_same_rows"] <= 1e-4, m
    assert m["Lhost_rel"] <= 1e-5 and m["Lfinal_vs_oracle_state"] <= 1e-5, m
    assert m["gpu_no_worse_than_host"], m
    if early_stop:
        assert np.mean(st.iters == res.iters) >= 0.99


def test_mu_one_is_the_main_refinement(jarq):
    lay = mu_layer(256, 40, 64, 3, drift=0.08, seed=9)
    dev = "cuda"
    hess = jarq.prepare(torch.as_tensor(lay.H, device=dev), lay.g)
    W = torch.as_tensor(lay.W, device=dev)
    Z = torch.as_tensor(lay.Z, device=dev)
    S1, Q1 = torch.as_tensor(lay.S0, device=dev).clone(), torch.as_tensor(lay.Q0, device=dev).clone()
    S2, Q2 = S1.clone(), Q1.clone()
    jarq.refine(hess, W, S1, Q1, Z, lay.bits, max_iters=3)
    jarq.refine_mu(hess, W, S2, Q2, Z, lay.bits, None, None, 1.0, lay.nu2, max_iters=3)
    assert torch.equal(S1, S2) and torch.equal(Q1, Q2)
    hess.close()


def test_mu_target_bad_arguments(jarq):
    lay = mu_layer(128, 8, 64, 3, seed=10)
    hess = jarq.prepare(lay.H, lay.g)
    for mu, nu2, K, XX in [(1.5, lay.nu2, lay.K, lay.XX), (-0.1, lay.nu2, lay.K, lay.XX),
                           (0.5, -1.0, lay.K, lay.XX), (0.5, float("inf"), lay.K, lay.XX),
                           (0.5, lay.nu2, None, lay.XX), (0.5, lay.nu2, lay.K, None)]:
        S, Q = lay.S0.copy(), lay.Q0.copy()
        st = jarq.refine_mu(hess, lay.W, S, Q, lay.Z, 3, K, XX, mu, nu2, max_iters=2,
                            raise_on_error=False)
        assert st.status == jarq.JARQ_ERR_ARG
        assert np.array_equal(S, lay.S0) and np.array_equal(Q, lay.Q0)
    # host buffers give the device result
    S, Q = lay.S0.copy(), lay.Q0.copy()
    jarq.refine_mu(hess, lay.W, S, Q, lay.Z, 3, lay.K, lay.XX, 0.5, lay.nu2, max_iters=2)
    Sd = torch.as_tensor(lay.S0, device="cuda").clone()
    Qd = torch.as_tensor(lay.Q0, device="cuda").clone()
    jarq.refine_mu(hess, torch.as_tensor(lay.W, device="cuda"), Sd, Qd,
                   torch.as_tensor(lay.Z, device="cuda"), 3, torch.as_tensor(lay.K, device="cuda"),
                   torch.as_tensor(lay.XX, device="cuda"), 0.5, lay.nu2, max_iters=2)
    assert np.array_equal(S, Sd.cpu().numpy()) and np.array_equal(Q, Qd.cpu().numpy())
    hess.close()


def test_mu_target_full_size_sampled_rows(jarq):
    """Llama-2-7B q_proj shape (4096 x 4096, g = 128, 3-bit, K = 10) on the
    mu = 0.5 target over 128 x 2048 drifted tokens: the CUDA path refines the
    whole layer, the oracle 32 seeded rows of it."""
    from synth.qep import mu_config_layer
    from types import SimpleNamespace
    lay, K, XX, nu2 = mu_config_layer("llama2_7b_q_proj_4096x4096_g128_w3", device="cuda")
    mu = 0.5
    hess = jarq.prepare(lay.H, lay.g)
    S, Q = lay.S0.clone(), lay.Q0.clone()
    st = jarq.refine_mu(hess, lay.W, S, Q, lay.Z, lay.bits, K, XX, mu, nu2, max_iters=lay.K,
                        early_stop=0)
    torch.cuda.synchronize()
    hess.close()
    rng = np.random.Generator(np.random.PCG64(321))
    rows = np.sort(rng.choice(lay.dout, 32, replace=False))
    cpu = lambda t: t.cpu().numpy()
    Hn, Kn, XXn = cpu(lay.H), cpu(K), cpu(XX)
    sub = SimpleNamespace(H=Hn, K=Kn, XX=XXn, W=cpu(lay.W)[rows], S0=cpu(lay.S0)[rows],
                          Q0=cpu(lay.Q0)[rows], Z=cpu(lay.Z)[rows], g=lay.g, bits=lay.bits)
    res, Wc, c = refine_mu(sub.H, sub.K, sub.XX, sub.W, sub.S0, sub.Q0, sub.Z, sub.bits, sub.g,
                           mu, nu2, Options(max_iters=lay.K, early_stop=False))
    s = SimpleNamespace(L_host=cpu(st.L_host)[rows], L_final=cpu(st.L_final)[rows])
    m = mu_compare(sub, mu, res, Wc, c, cpu(S)[rows], cpu(Q)[rows], s)
    print(m)
    assert m["codes_same"] >= 0.999, m
    assert m["S_rel_max_same_rows"] <= 1e-4 and m["F_rel_max_same_rows"] <= 1e-4, m
    assert m["Lhost_rel"] <= 1e-5 and m["Lfinal_vs_oracle_state"] <= 1e-5, m
    assert m["gpu_no_worse_than_host"], m
