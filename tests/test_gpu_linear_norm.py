"""sq_linear_norm: the pre-norm projection in one call.  It must equal
sq_rmsnorm followed by sq_linear_ex bit for bit on both engines (the GEMV
normalises while staging, in the standalone kernel's arithmetic order; the
tensor-core path runs that kernel first), and the fp64 oracle
(rmsnorm, then the linear over the dequantised weights) within the linear
tolerance."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq

from gpu_util import assert_close, dev, dev_to_f64, f16_to_dev

pytestmark = pytest.mark.gpu
EPS = 1e-6
KINDS = {"fp16": sq.SQ_W_FP16, "int4": sq.SQ_W_INT4, "fp8": sq.SQ_W_FP8}


def _weights(kind, N, K, seed):
    """Device weights of the variant and their fp64 dequantised values, both
    from the oracle's quantiser (no oracle input comes from the GPU)."""
    rng = np.random.default_rng(seed)
    w16 = (rng.standard_normal((N, K)) * 0.02).astype(np.float16)
    if kind == "fp16":
        return f16_to_dev(w16), None, w16.astype(np.float64)
    if kind == "int4":
        c, s = oracle.quantize_int4(w16.view(np.uint16))
        return torch.from_numpy(c).to(dev()), f16_to_dev(s.view(np.float16)), oracle.dequant_int4(c, s, K)
    c, s = oracle.quantize_fp8(w16.view(np.uint16))
    return torch.from_numpy(c).to(dev()), torch.from_numpy(s).to(dev()), oracle.dequant_fp8(c, s)


@pytest.mark.parametrize("kind", ["fp16", "int4", "fp8"])
@pytest.mark.parametrize("M,N,K,epi", [
    (1, 2048, 1536, sq.SQ_EPI_NONE),          # q/k/v of the 1.5B shape
    (1, 17920, 1536, sq.SQ_EPI_SILU_GATE),    # gate/up
    (1, 9000, 896, sq.SQ_EPI_NONE),           # INT4: many 16-row tiles, register-operand tensor path
    (2, 640, 896, sq.SQ_EPI_NONE),
    (5, 2048, 1536, sq.SQ_EPI_NONE),          # verify rows
    (16, 1024, 3584, sq.SQ_EPI_SILU_GATE),
    (48, 512, 1536, sq.SQ_EPI_NONE),          # tensor-core rows
])
def test_linear_norm_equals_rmsnorm_then_linear(kind, M, N, K, epi):
    rng = np.random.default_rng(M * 7 + N)
    x16 = (rng.standard_normal((M, K)) * 3).astype(np.float16)
    g16 = (1 + 0.1 * rng.standard_normal(K)).astype(np.float16)
    x, g = f16_to_dev(x16), f16_to_dev(g16)
    w, s, wd = _weights(kind, N, K, M + N + K)
    ncols = N // 2 if epi == sq.SQ_EPI_SILU_GATE else N
    wk = KINDS[kind]
    h = torch.empty(M, K, dtype=torch.float16, device=dev())
    y1 = torch.empty(M, ncols, dtype=torch.float16, device=dev())
    sq.sq_rmsnorm(x, g, EPS, h)
    sq.sq_linear_ex(wk, h, w, s, None, None, epi, y1)
    xn = torch.empty(M, K, dtype=torch.float16, device=dev())
    y2 = torch.empty(M, ncols, dtype=torch.float16, device=dev())
    sq.sq_linear_norm(wk, x, g, EPS, xn, w, s, None, None, epi, y2)
    assert sq.sq_check() == 0
    assert torch.equal(y1.view(torch.int16), y2.view(torch.int16)), sq.sq_linear_path(wk, M, N, K, epi)
    hn = oracle.rmsnorm(x16.astype(np.float64), g16.astype(np.float64), EPS)
    ref = oracle.linear(hn, wd)
    if epi == sq.SQ_EPI_SILU_GATE:
        ref = oracle.silu_gate(ref[:, :ncols], ref[:, ncols:])
    assert_close(dev_to_f64(y2), ref, f"{kind} M={M}")


def test_linear_norm_with_residual_epilogue():
    rng = np.random.default_rng(5)
    M, N, K = 1, 1536, 8960
    x = f16_to_dev((rng.standard_normal((M, K))).astype(np.float16))
    g = f16_to_dev((1 + 0.1 * rng.standard_normal(K)).astype(np.float16))
    r = f16_to_dev((rng.standard_normal((M, N))).astype(np.float16))
    w, s, _ = _weights("int4", N, K, 9)
    h = torch.empty(M, K, dtype=torch.float16, device=dev())
    y1 = torch.empty(M, N, dtype=torch.float16, device=dev())
    sq.sq_rmsnorm(x, g, EPS, h)
    sq.sq_linear_ex(sq.SQ_W_INT4, h, w, s, None, r, sq.SQ_EPI_RESIDUAL, y1)
    y2 = r.clone()
    xn = torch.empty_like(h)
    sq.sq_linear_norm(sq.SQ_W_INT4, x, g, EPS, xn, w, s, None, y2, sq.SQ_EPI_RESIDUAL, y2)
    assert sq.sq_check() == 0
    assert torch.equal(y1.view(torch.int16), y2.view(torch.int16))


def test_linear_norm_rejects_aliased_scratch():
    x = torch.zeros(1, 256, dtype=torch.float16, device=dev())
    g = torch.ones(256, dtype=torch.float16, device=dev())
    w = torch.zeros(64, 256, dtype=torch.float16, device=dev())
    y = torch.empty(1, 64, dtype=torch.float16, device=dev())
    with pytest.raises(sq.SQError):
        sq.sq_linear_norm(sq.SQ_W_FP16, x, g, EPS, x, w, None, None, None, sq.SQ_EPI_NONE, y)
