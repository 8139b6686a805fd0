"""Full-size layers: the CUDA path refines the whole layer; the oracle
refines a seeded sample of its rows (rows are independent, Sec. 3.3), and
the two are compared on those rows.  Same bar as the small-layer tests.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

from oracle import Options, prepare_hessian, refine_layer  # noqa: E402
from synth import CONFIGS, Layer, config_layer  # noqa: E402
from tests.parity import compare_final, gpu_refine, lockstep  # noqa: E402

N_SAMPLE = 48


def sample_rows(dout, n, seed=123):
    rng = np.random.default_rng(seed)
    return np.sort(rng.choice(dout, size=min(n, dout), replace=False))


def to_np(lay):
    return Layer(lay.name, lay.W.cpu().numpy(), lay.H.cpu().numpy(), lay.S0.cpu().numpy(),
                 lay.Q0.cpu().numpy(), lay.Z.cpu().numpy(), lay.bits, lay.g, lay.K)


def sub_layer(lay_np, rows):
    return Layer(lay_np.name, lay_np.W[rows], lay_np.H, lay_np.S0[rows], lay_np.Q0[rows],
                 lay_np.Z[rows], lay_np.bits, lay_np.g, lay_np.K)


@pytest.mark.parametrize("name", [
    "llama2_7b_q_proj_4096x4096_g128_w3",
    "llama2_7b_q_proj_4096x4096_g64_w3",      # 64 groups per row
    "llama2_7b_down_proj_4096x11008_g128_w4",
    "llama3_8b_gate_proj_14336x4096_g128_w3",
])
def test_full_layer_sampled_rows(name):
    from paper_2609_38599_gb300 import jarq
    lay = config_layer(name, device="cuda")
    K = lay.K
    hess = jarq.prepare(lay.H, lay.g)
    S = lay.S0.clone()
    Q = lay.Q0.clone()
    st = jarq.refine(hess, lay.W, S, Q, lay.Z, lay.bits, max_iters=K, early_stop=0)
    torch.cuda.synchronize()
    hess.close()
    lay_np = to_np(lay)
    rows = sample_rows(lay.dout, N_SAMPLE)
    sub = sub_layer(lay_np, rows)
    prep = prepare_hessian(sub.H, sub.g)
    res = refine_layer(prep, sub.W, sub.S0, sub.Q0, sub.Z, sub.bits,
                       Options(max_iters=K, early_stop=False))
    stats = {"L_host": st.L_host.cpu().numpy()[rows], "L_final": st.L_final.cpu().numpy()[rows]}
    m = compare_final(sub, prep, res, S.cpu().numpy()[rows], Q.cpu().numpy()[rows], stats)
    print(name, m)
    assert m["Lhost_rel"] <= 1e-5 and m["Lfinal_vs_oracle_state"] <= 1e-5, m
    assert m["S_rel_max_same_rows"] <= 1e-4 and m["F_rel_max_same_rows"] <= 1e-4, m
    assert m["F_rel_all"] <= 1e-4, m
    assert m["gpu_no_worse_than_host"], m
    assert m["codes_same"] >= 0.999, m
    # format: whole layer
    assert int(Q.max()) <= (1 << lay.bits) - 1


def test_full_layer_early_stop_q_proj():
    """The q_proj layer with the early stop on (App. E "Early stopping",
    tau_rel = tau_abs = 1e-5): the whole layer on the GPU, 48 seeded rows on
    the oracle; the same bar, and the iteration counts must agree."""
    from paper_2609_38599_gb300 import jarq
    name = "llama2_7b_q_proj_4096x4096_g128_w3"
    lay = config_layer(name, device="cuda")
    hess = jarq.prepare(lay.H, lay.g)
    S = lay.S0.clone()
    Q = lay.Q0.clone()
    st = jarq.refine(hess, lay.W, S, Q, lay.Z, lay.bits, max_iters=lay.K, early_stop=1)
    torch.cuda.synchronize()
    hess.close()
    rows = sample_rows(lay.dout, N_SAMPLE, seed=321)
    sub = sub_layer(to_np(lay), rows)
    prep = prepare_hessian(sub.H, sub.g)
    res = refine_layer(prep, sub.W, sub.S0, sub.Q0, sub.Z, sub.bits,
                       Options(max_iters=lay.K, early_stop=True))
    stats = {"L_host": st.L_host.cpu().numpy()[rows], "L_final": st.L_final.cpu().numpy()[rows]}
    m = compare_final(sub, prep, res, S.cpu().numpy()[rows], Q.cpu().numpy()[rows], stats)
    iters = st.iters.cpu().numpy()[rows]
    m["iters_agree"] = float(np.mean(iters == res.iters))
    print(name, "early stop", m, "iters", np.bincount(iters))
    assert m["Lhost_rel"] <= 1e-5 and m["Lfinal_vs_oracle_state"] <= 1e-5, m
    assert m["S_rel_max_same_rows"] <= 1e-4 and m["F_rel_max_same_rows"] <= 1e-4, m
    assert m["F_rel_all"] <= 1e-4, m
    assert m["gpu_no_worse_than_host"], m
    assert m["codes_same"] >= 0.999, m
    # a stop decided within rounding of the threshold counts as a near-tie;
    # none is expected on 48 rows
    assert m["iters_agree"] >= 0.97, m


@pytest.mark.parametrize("name,n", [("llama2_7b_q_proj_4096x4096_g128_w3", 24),
                                    ("llama2_7b_down_proj_4096x11008_g128_w4", 12),
                                    ("llama3_8b_gate_proj_14336x4096_g128_w3", 12)])
def test_lockstep_sampled_rows(name, n):
    """Both sides step one iteration at a time from the oracle's state; every
    difference must start at a near-tie of the oracle's own values."""
    lay = config_layer(name, device="cuda")
    sub = sub_layer(to_np(lay), sample_rows(lay.dout, n, seed=7))

    def step(S, Q):
        S2, Q2, _ = gpu_refine(sub, 1, S=S, Q=Q)
        return S2, Q2

    recs = lockstep(sub, lay.K, step)
    print(recs)


def test_lockstep_decoder_block_one_layer_per_hessian():
    """Near-tie tracing on the decoder block: one layer on each of its three
    Hessians (q_proj on the attention input, o_proj, down_proj), 6 seeded
    rows each, stepped one iteration at a time from the oracle's state."""
    from synth import block_layers
    hs, layers = block_layers(device="cuda")
    seen = set()
    for idx, (hkey, lay) in enumerate(layers):
        if hkey in seen:
            continue
        seen.add(hkey)
        sub = sub_layer(to_np(lay), sample_rows(lay.dout, 6, seed=300 + idx))

        def step(S, Q, sub=sub):
            S2, Q2, _ = gpu_refine(sub, 1, S=S, Q=Q)
            return S2, Q2

        recs = lockstep(sub, lay.K, step)
        print(lay.name, recs)
    assert len(seen) == 3


def test_decoder_block_sampled_rows():
    """The Llama-2-7B decoder block: three Hessians, each prepared once, and
    the seven layers refined on them (q/k/v/gate/up share the attention-input
    H); every layer is compared with the oracle on a seeded sample of rows."""
    from paper_2609_38599_gb300 import jarq
    from synth import block_layers
    hs, layers = block_layers(device="cuda")
    hess = {k: jarq.prepare(h, 128) for k, h in hs.items()}
    preps = {}
    for idx, (hkey, lay) in enumerate(layers):
        S = lay.S0.clone()
        Q = lay.Q0.clone()
        st = jarq.refine(hess[hkey], lay.W, S, Q, lay.Z, lay.bits, max_iters=lay.K, early_stop=0)
        torch.cuda.synchronize()
        rows = sample_rows(lay.dout, 8, seed=200 + idx)
        sub = sub_layer(to_np(lay), rows)
        if hkey not in preps:
            preps[hkey] = prepare_hessian(sub.H, sub.g)
        prep = preps[hkey]
        res = refine_layer(prep, sub.W, sub.S0, sub.Q0, sub.Z, sub.bits,
                           Options(max_iters=lay.K, early_stop=False))
        stats = {"L_host": st.L_host.cpu().numpy()[rows], "L_final": st.L_final.cpu().numpy()[rows]}
        m = compare_final(sub, prep, res, S.cpu().numpy()[rows], Q.cpu().numpy()[rows], stats)
        print(lay.name, m)
        assert m["Lhost_rel"] <= 1e-5 and m["Lfinal_vs_oracle_state"] <= 1e-5, (lay.name, m)
        assert m["S_rel_max_same_rows"] <= 1e-4 and m["F_rel_max_same_rows"] <= 1e-4, (lay.name, m)
        assert m["F_rel_all"] <= 1e-4, (lay.name, m)
        assert m["gpu_no_worse_than_host"], (lay.name, m)
        assert m["codes_same"] >= 0.999, (lay.name, m)
    for h in hess.values():
        h.close()
