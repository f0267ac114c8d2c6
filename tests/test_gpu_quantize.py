"""GPU parity: sq_quantize (Sec. III-A.1 Q4 = f(W16,4), Sec. III-A.2 Q8 =
f(W16,8)) against the oracle, bit-exact codes and scales."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq
from paper_2609_21704_gb300 import synth
from paper_2609_21704_gb300.shapes import QWEN25_1P5B, QWEN25_7B

from gpu_util import bits16, dev, f16_to_dev

pytestmark = pytest.mark.gpu


def _quant_gpu(w: np.ndarray, kind):
    return _quant_gpu_dev(f16_to_dev(w), kind)


def _quant_gpu_dev(wt, kind):
    N, K = wt.shape
    cb, sb = sq.sq_quantized_bytes(kind, N, K)
    codes = torch.empty(cb, dtype=torch.uint8, device=dev())
    if kind == sq.SQ_INT4_G128:
        scales = torch.empty(sb // 2, dtype=torch.float16, device=dev())
    else:
        scales = torch.empty(sb // 4, dtype=torch.float32, device=dev())
    sq.sq_quantize(wt, kind, codes, scales)
    assert sq.sq_check() == 0
    return codes, scales


def _check_int4(w, codes, scales, rows=None):
    N, K = w.shape
    c = codes.cpu().numpy().reshape(N, K // 2)
    s = bits16(scales).reshape(N, K // 128)
    if rows is not None:
        w, c, s = w[rows], c[rows], s[rows]
    oc, os_ = oracle.quantize_int4(w.view(np.uint16))
    assert np.array_equal(c, oc)
    assert np.array_equal(s, os_)


def _check_fp8(w, codes, scales, rows=None):
    N, K = w.shape
    c = codes.cpu().numpy().reshape(N, K)
    s = scales.cpu().numpy()
    if rows is not None:
        w, c, s = w[rows], c[rows], s[rows]
    oc, os_ = oracle.quantize_fp8(w.view(np.uint16))
    assert np.array_equal(c, oc)
    assert np.array_equal(s.view(np.uint32), os_.view(np.uint32))


def _edge_matrix(K):
    w = synth.weights_fp16(5, 24, K).copy()
    w[0] = 0                                   # all-zero rows / groups
    w[1, :] = np.float16(-0.0)
    w[2, :] = np.float16(2.0 ** -24)           # smallest subnormal: INT4 scale fallback
    w[3, ::3] = np.float16(3 * 2.0 ** -24)
    w[4, :] = np.float16(65504.0)              # largest finite
    w[5, 7] = np.float16(-65504.0)
    w[6] = (np.arange(K) % 17 - 8).astype(np.float16)  # ties at scale 8/7
    w[7] = np.float16(0.5) * (np.arange(K) % 2 * 2 - 1)
    return w


@pytest.mark.parametrize("N,K", [(1, 128), (64, 896), (257, 1536), (33, 4864)])
def test_int4_bitexact_small(N, K):
    w = synth.weights_fp16(N * 7 + K, N, K)
    _check_int4(w, *_quant_gpu(w, sq.SQ_INT4_G128))


@pytest.mark.parametrize("N,K", [(1, 16), (64, 896), (257, 1536), (33, 4864), (5, 18944)])
def test_fp8_bitexact_small(N, K):
    w = synth.weights_fp16(N * 11 + K, N, K)
    _check_fp8(w, *_quant_gpu(w, sq.SQ_FP8_E4M3_ROW))


@pytest.mark.parametrize("K", [128, 1024])
def test_edge_values_bitexact(K):
    w = _edge_matrix(K)
    _check_int4(w, *_quant_gpu(w, sq.SQ_INT4_G128))
    _check_fp8(w, *_quant_gpu(w, sq.SQ_FP8_E4M3_ROW))


@pytest.mark.parametrize("shape", [QWEN25_1P5B.lm_head(), QWEN25_7B.projections()[3],
                                   QWEN25_7B.projections()[2]])
def test_full_size_sampled_rows(shape):
    _, N, K = shape
    wt = synth.weights_fp16_device(N + K, N, K, dev())
    rows = np.unique(np.concatenate([[0, 1, N - 1], np.random.default_rng(N).integers(0, N, 96)]))
    w_rows = bits16(wt[torch.from_numpy(rows).to(dev())]).view(np.float16)
    for kind, check in ((sq.SQ_INT4_G128, _check_int4), (sq.SQ_FP8_E4M3_ROW, _check_fp8)):
        codes, scales = _quant_gpu_dev(wt, kind)
        cb = codes.view(N, -1)[torch.from_numpy(rows).to(dev())].reshape(-1)
        sb = scales.view(N, -1)[torch.from_numpy(rows).to(dev())].reshape(-1)
        check(w_rows, cb, sb)


def test_nonfinite_weight_sets_status_bit():
    w = synth.weights_fp16(9, 4, 256)
    w[2, 77] = np.float16(np.inf)
    wt = f16_to_dev(w)
    codes = torch.empty(4 * 128, dtype=torch.uint8, device=dev())
    scales = torch.empty(8, dtype=torch.float16, device=dev())
    sq.sq_quantize(wt, sq.SQ_INT4_G128, codes, scales)
    assert sq.sq_check() & sq.SQ_DEV_NONFINITE_WEIGHT
    assert sq.sq_check() == 0  # reading clears the word
    c8 = torch.empty(4 * 256, dtype=torch.uint8, device=dev())
    s8 = torch.empty(4, dtype=torch.float32, device=dev())
    sq.sq_quantize(wt, sq.SQ_FP8_E4M3_ROW, c8, s8)
    assert sq.sq_check() & sq.SQ_DEV_NONFINITE_WEIGHT


def test_runs_on_sm_103a():
    """The library carries sm_103a machine code only (no PTX to fall back
    on), so a kernel that ran and gave bit-exact codes ran as sm_103a code
    on a compute capability 10.3 device."""
    assert torch.cuda.get_device_capability(dev()) == (10, 3)
    w = synth.weights_fp16(3, 16, 128)
    codes = torch.empty(16, 64, dtype=torch.uint8, device=dev())
    scales = torch.empty(16, 1, dtype=torch.float16, device=dev())
    sq.sq_quantize(f16_to_dev(w), sq.SQ_INT4_G128, codes, scales)
    c, _ = oracle.quantize_int4(w.view(np.uint16))
    assert np.array_equal(codes.cpu().numpy(), c)
