"""GPU parity: the tcgen05 tensor-core linear layer (M >= 16 activation
rows with fp16 weights: Sec. III-D.3 verify pass at B * (K+1) rows) against
the fp64 oracle.  Covers ragged N (not a multiple of the 128-row tile) and
ragged K (not a multiple of the 64-wide stage), split-K over clusters, the
SiLU-gate / residual / bias epilogues and a full-size 7B projection."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq
from paper_2609_21704_gb300 import synth
from paper_2609_21704_gb300.shapes import QWEN25_7B

from gpu_util import assert_close, bits16, dev, dev_to_f64, f16_to_dev

pytestmark = pytest.mark.gpu


def _tc(x, w, N_out, bias=None, residual=None, epi=sq.SQ_EPI_NONE, y=None):
    if y is None:
        y = torch.empty(x.shape[0], N_out, dtype=torch.float16, device=dev())
    sq.sq_linear_ex(sq.SQ_W_FP16, x, w, None, bias, residual, epi, y)
    assert sq.sq_check() == 0
    return y


@pytest.mark.parametrize("M", [16, 17, 32, 48, 100, 144, 256])
@pytest.mark.parametrize("N,K", [(128, 64), (200, 1000), (1536, 1536), (384, 8960)])
def test_tc_matches_oracle(M, N, K):
    w = synth.weights_fp16(M + N + K, N, K)
    x = synth.activations_fp16(M * 3 + K, M, K)
    y = _tc(f16_to_dev(x), f16_to_dev(w), N)
    assert_close(dev_to_f64(y), oracle.linear(x.astype(np.float64), w.astype(np.float64)), f"M={M} N={N} K={K}")


@pytest.mark.parametrize("M", [16, 48])
def test_tc_silu_bias_residual(M):
    I, K = 320, 1536
    w = synth.weights_fp16(21, 2 * I, K)
    x = synth.activations_fp16(22, M, K)
    b = synth.fp16_normal(23, (2 * I,), 0.5)
    y = _tc(f16_to_dev(x), f16_to_dev(w), I, bias=f16_to_dev(b), epi=sq.SQ_EPI_SILU_GATE)
    full = oracle.linear(x.astype(np.float64), w.astype(np.float64), b.astype(np.float64))
    assert_close(dev_to_f64(y), oracle.silu_gate(full[:, :I], full[:, I:]), "silu")
    N = 600
    w2 = synth.weights_fp16(24, N, K)
    r = synth.fp16_normal(25, (M, N), 1.0)
    yr = f16_to_dev(r)
    _tc(f16_to_dev(x), f16_to_dev(w2), N, residual=yr, epi=sq.SQ_EPI_RESIDUAL, y=yr)
    ref = oracle.linear(x.astype(np.float64), w2.astype(np.float64)) + r.astype(np.float64)
    assert_close(dev_to_f64(yr), ref, "residual")


def test_tc_repeatable_bit_for_bit():
    M, N, K = 48, 3584, 3584
    w = f16_to_dev(synth.weights_fp16(31, N, K))
    x = f16_to_dev(synth.activations_fp16(32, M, K))
    assert torch.equal(_tc(x, w, N), _tc(x, w, N))


@pytest.mark.parametrize("M", [48, 144])
def test_tc_full_size_down_proj_7b_sampled(M):
    _, N, K = QWEN25_7B.projections()[3]
    wt = synth.weights_fp16_device(41, N, K, dev())
    xt = synth.activations_fp16_device(42, M, K, dev())
    y = _tc(xt, wt, N)
    cols = np.unique(np.concatenate([[0, N - 1], np.random.default_rng(M).integers(0, N, 62)]))
    w_rows = bits16(wt[torch.from_numpy(cols).to(dev())]).view(np.float16).astype(np.float64)
    x64 = bits16(xt).view(np.float16).astype(np.float64)
    assert_close(dev_to_f64(y)[:, cols], oracle.linear(x64, w_rows), f"7B down M={M}")
