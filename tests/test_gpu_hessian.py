"""Calibration-Hessian accumulation on the tensor cores (through the C ABI)
against the float64 oracle ``accumulate_hessian``.

Bars:
* integer-valued fp16 activations whose sums stay below 2^24: every product
  and every partial sum is exact in float32, so the result must be bit-exact
  (this also fixes indexing: tiles, mirrors, ragged edges, each element
  written exactly once);
* general activations: the CUDA path sums in float32 (the tensor cores over
  blocks of 512 tokens, i.e. 32 MMAs of 16 tokens, then the blocks in
  registers) and rounds once into H.  Counting every MMA as two roundings
  (it may truncate) and every block addition as one, the error of element
  (i, j) is at most gamma * sum_t |x_ti x_tj| + 2^-24 |H_ij| with
  gamma = (2 * 32 + blocks + 1) * 2^-23.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

from oracle import accumulate_hessian  # noqa: E402
from synth import activations_np, config_activations, integer_activations_np  # noqa: E402

SEG = 512


@pytest.fixture(scope="module")
def jarq():
    from paper_2609_38599_gb300 import jarq as mod
    return mod


def gamma(n):
    blocks = max(1, -(-n // SEG))
    return (2 * (SEG // 16) + blocks + 1) * 2.0 ** -23


@pytest.mark.parametrize("n,d", [(1, 8), (63, 200), (1000, 264), (3000, 520), (2100, 1024),
                                 (20000, 640)])
def test_integer_activations_bit_exact(jarq, n, d):
    X = integer_activations_np(n, d, amax=8, seed=n + d)
    rng = np.random.Generator(np.random.PCG64(d))
    H0 = rng.integers(-1000, 1000, size=(d, d)).astype(np.float32)   # not symmetric
    ref = accumulate_hessian(X, H0.astype(np.float64))
    assert np.abs(ref).max() < 2 ** 24
    H = torch.as_tensor(H0, device="cuda").clone()
    jarq.accumulate_hessian(torch.as_tensor(X, device="cuda"), H)
    np.testing.assert_array_equal(H.cpu().numpy(), ref.astype(np.float32))


def test_streamed_batches_and_scale_bit_exact(jarq):
    d = 392
    X = integer_activations_np(5000, d, amax=6, seed=11)
    Xd = torch.as_tensor(X, device="cuda")
    H = torch.zeros(d, d, device="cuda")
    for a, b in [(0, 64), (64, 1100), (1100, 1101), (1101, 5000)]:
        jarq.accumulate_hessian(Xd[a:b].contiguous(), H, scale=0.5)
    ref = accumulate_hessian(X, scale=0.5)
    np.testing.assert_array_equal(H.cpu().numpy(), ref.astype(np.float32))
    # exactly symmetric
    Hn = H.cpu().numpy()
    np.testing.assert_array_equal(Hn, Hn.T)


@pytest.mark.parametrize("n,d", [(4096, 384), (5000, 520)])
def test_float_activations_within_bound(jarq, n, d):
    X = activations_np(n, d, rank=8, n_out=3, seed=n + d)
    ref = accumulate_hessian(X)
    absdot = accumulate_hessian(np.abs(X))
    H = jarq.accumulate_hessian(torch.as_tensor(X, device="cuda")).cpu().numpy()
    err = np.abs(H.astype(np.float64) - ref)
    bound = gamma(n) * absdot + 2.0 ** -24 * np.abs(ref)
    print("max err / bound", float((err / bound).max()),
          "max rel err", float((err / np.abs(ref).clip(1e-30)).max()))
    assert np.all(err <= bound)
    np.testing.assert_array_equal(H, H.T)


def test_zero_tokens_and_bad_arguments(jarq):
    from paper_2609_38599_gb300.jarq import JarqError, JARQ_ERR_ARG, _lib
    import ctypes
    d = 64
    H = torch.full((d, d), 3.0, device="cuda")
    X = torch.zeros(0, d, dtype=torch.float16, device="cuda")
    jarq.accumulate_hessian(X, H)
    assert bool((H == 3.0).all())
    # d not a multiple of 8
    X12 = torch.ones(16, 12, dtype=torch.float16, device="cuda")
    with pytest.raises(JarqError) as ei:
        jarq.accumulate_hessian(X12)
    assert ei.value.status == JARQ_ERR_ARG
    # X not 16-byte aligned
    buf = torch.ones(16 * 64 + 1, dtype=torch.float16, device="cuda")
    Xm = buf[1:].view(16, 64)
    with pytest.raises(JarqError) as ei:
        jarq.accumulate_hessian(Xm, H)
    assert ei.value.status == JARQ_ERR_ARG
    assert bool((H == 3.0).all())
    # H not 16-byte aligned
    hbuf = torch.zeros(d * d + 1, device="cuda")
    with pytest.raises(JarqError) as ei:
        jarq.accumulate_hessian(torch.ones(16, d, dtype=torch.float16, device="cuda"),
                                hbuf[1:].view(d, d))
    assert ei.value.status == JARQ_ERR_ARG
    # host H
    Hh = np.zeros((d, d), np.float32)
    Xd = torch.ones(16, d, dtype=torch.float16, device="cuda")
    st = _lib.jarq_accumulate_hessian(ctypes.c_void_p(Xd.data_ptr()), 16, d, 1.0,
                                      ctypes.c_void_p(Hh.ctypes.data), None)
    assert st == JARQ_ERR_ARG
    # non-finite scale
    st = _lib.jarq_accumulate_hessian(ctypes.c_void_p(Xd.data_ptr()), 16, d, float("nan"),
                                      ctypes.c_void_p(H.data_ptr()), None)
    assert st == JARQ_ERR_ARG


def test_full_size_attention_input_sampled(jarq):
    """The Llama-2-7B attention input (d = 4096) over 128 x 2048 tokens, in
    one call; 96 sampled features (all pairs among them) against the
    oracle."""
    X = config_activations("llama2_7b_attn_in_4096_n262144", device="cuda")
    n, d = X.shape
    H = jarq.accumulate_hessian(X)
    torch.cuda.synchronize()
    rng = np.random.Generator(np.random.PCG64(99))
    idx = np.sort(np.concatenate([[0, d - 1],
                                  rng.choice(np.arange(1, d - 1), 94, replace=False)]))
    # the heaviest channels (the outliers) are part of the sample
    norms = X.float().pow(2).sum(0)
    top = torch.topk(norms, 8).indices.cpu().numpy()
    idx = np.unique(np.concatenate([idx, top]))
    it = torch.as_tensor(idx, device="cuda")
    Xs = X.index_select(1, it).cpu().numpy()
    ref = accumulate_hessian(Xs)
    absdot = accumulate_hessian(np.abs(Xs))
    Hs = H.index_select(0, it).index_select(1, it).cpu().numpy().astype(np.float64)
    err = np.abs(Hs - ref)
    bound = gamma(n) * absdot + 2.0 ** -24 * np.abs(ref)
    print("full size: max err / bound", float((err / bound).max()),
          "max rel err (diag)", float((err.diagonal() / ref.diagonal()).max()))
    assert np.all(err <= bound)
    Hn = H.cpu().numpy()
    assert np.array_equal(Hn, Hn.T)
    del X, H
    torch.cuda.empty_cache()


def test_full_size_down_proj_input_sampled(jarq):
    """The down_proj input (d = 11008, 1892 tiles) over 64 x 2048 tokens, in
    one call; 64 sampled features against the oracle."""
    X = config_activations("llama2_7b_down_in_11008_n131072", device="cuda")
    n, d = X.shape
    H = jarq.accumulate_hessian(X)
    torch.cuda.synchronize()
    rng = np.random.Generator(np.random.PCG64(7))
    idx = np.sort(np.concatenate([[0, d - 1], rng.choice(np.arange(1, d - 1), 62, replace=False)]))
    it = torch.as_tensor(idx, device="cuda")
    Xs = X.index_select(1, it).cpu().numpy()
    ref = accumulate_hessian(Xs)
    absdot = accumulate_hessian(np.abs(Xs))
    Hs = H.index_select(0, it).index_select(1, it).cpu().numpy().astype(np.float64)
    err = np.abs(Hs - ref)
    bound = gamma(n) * absdot + 2.0 ** -24 * np.abs(ref)
    print("down_in: max err / bound", float((err / bound).max()))
    assert np.all(err <= bound)
    Hn = H.cpu().numpy()
    assert np.array_equal(Hn, Hn.T)
    del X, H
    torch.cuda.empty_cache()
