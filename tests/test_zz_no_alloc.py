"""The allocation-free objective entry point matches the regular one.

jarq_objective_noalloc serves callers that must not allocate device memory
when they ask for the objective (processes that reserve all device memory at
start-up, or that cannot afford an allocation's synchronisation).  Its
scratch is one static device array shared by every call, so the test calls
it twice in a row with different states and checks each result against
jarq_objective and against the float64 oracle's objective of the same
state, and that the device's free memory does not move during a call.  This
file is collected last so that a run stopping at the first failure has
already run every other test; it also passes when run alone.
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]


def _noalloc(J, hess, W, S, Q, Z, bits, F):
    lib = J.library()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return lib.jarq_objective_noalloc(hess.handle, W.data_ptr(), S.data_ptr(), Q.data_ptr(),
                                      Z.data_ptr(), int(W.shape[0]), int(bits), F.data_ptr(),
                                      stream)


def test_noalloc_objective_matches_regular_entry_point_twice():
    from paper_2609_38599_gb300 import jarq as J
    from synth import small_layer
    lay = small_layer(384, 200, 128, 3, seed=41)
    dev = "cuda"
    hess = J.prepare(torch.as_tensor(lay.H, device=dev), lay.g)
    W = torch.as_tensor(lay.W, device=dev)
    Z = torch.as_tensor(lay.Z, device=dev)
    states = [(torch.as_tensor(lay.S0, device=dev), torch.as_tensor(lay.Q0, device=dev))]
    # a second, different state: refined scales and codes
    S2 = states[0][0].clone()
    Q2 = states[0][1].clone()
    J.refine(hess, W, S2, Q2, Z, lay.bits, max_iters=2)
    states.append((S2, Q2))
    from oracle import objective, prepare_hessian
    prep = prepare_hessian(lay.H, lay.g)
    F_bufs = [torch.full((lay.dout,), float("nan"), dtype=torch.float64, device=dev)
              for _ in states]
    # warm-up: the first call on a device may load the library's module,
    # which places the static array on the GPU
    assert _noalloc(J, hess, W, *states[0], Z, lay.bits, F_bufs[0]) == J.JARQ_OK
    torch.cuda.synchronize()
    for (S, Q), F in zip(states, F_bufs):   # two calls in a row
        F_ref = J.objective(hess, W, S, Q, Z, lay.bits)
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        st = _noalloc(J, hess, W, S, Q, Z, lay.bits, F)
        free1 = torch.cuda.mem_get_info()[0]
        assert st == J.JARQ_OK, J.status_string(st)
        # no device allocation during the call
        assert free1 == free0, (free0, free1)
        np.testing.assert_allclose(F.cpu().numpy(), F_ref.cpu().numpy(), rtol=1e-12, atol=0)
        # and the value itself: the oracle's float64 objective of the same state
        F_orc = objective(prep, lay.W, S.cpu().numpy().astype(np.float64),
                          Q.cpu().numpy(), lay.Z)
        np.testing.assert_allclose(F.cpu().numpy(), F_orc, rtol=1e-5, atol=0)
    hess.close()


def test_noalloc_rejects_host_buffers_and_oversized_layers():
    from paper_2609_38599_gb300 import jarq as J
    from synth import small_layer
    lay = small_layer(256, 16, 128, 3, seed=42)
    hess = J.prepare(torch.as_tensor(lay.H, device="cuda"), lay.g)
    lib = J.library()
    F = np.zeros(lay.dout)
    st = lib.jarq_objective_noalloc(hess.handle, lay.W.ctypes.data, lay.S0.ctypes.data,
                                    lay.Q0.ctypes.data, lay.Z.ctypes.data, lay.dout, 3,
                                    F.ctypes.data, None)
    assert st == J.JARQ_ERR_ARG
    hess.close()
    # 2048 x 1024 padded elements exceed the 2^20 limit
    big = small_layer(2048, 1024, 128, 3, seed=43, rank=8, tokens=4096)
    hb = J.prepare(torch.as_tensor(big.H, device="cuda"), big.g)
    t = lambda a: torch.as_tensor(a, device="cuda")
    Fb = torch.zeros(big.dout, dtype=torch.float64, device="cuda")
    st = _noalloc(J, hb, t(big.W), t(big.S0), t(big.Q0), t(big.Z), 3, Fb)
    assert st == J.JARQ_ERR_ARG
    hb.close()
