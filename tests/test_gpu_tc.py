"""GPU parity: the tcgen05 tensor-core linear layer (Sec. III-D.3 verify
pass at B * (K+1) rows, and the draft pass at B rows) against the fp64
oracle: M >= 16 rows with fp16, FP8 and INT4 weights, and the 3..15-row
calls routed to it (rows padded with zeros).  Covers ragged N (not a
multiple of the 128-row tile) and ragged K (not a multiple of the 64-wide
stage), split-K over clusters, the SiLU-gate / residual / bias epilogues and
full-size 7B projections."""
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


def _quant_variant(kind, w):
    N, K = w.shape
    if kind == "int4":
        c, s = oracle.quantize_int4(w.view(np.uint16))
        return torch.from_numpy(c).to(dev()), f16_to_dev(s.view(np.float16)), oracle.dequant_int4(c, s, K)
    c, s = oracle.quantize_fp8(w.view(np.uint16))
    return torch.from_numpy(c).to(dev()), torch.from_numpy(s).to(dev()), oracle.dequant_fp8(c, s)


WKQ = {"int4": sq.SQ_W_INT4, "fp8": sq.SQ_W_FP8}


@pytest.mark.parametrize("kind", ["int4", "fp8"])
@pytest.mark.parametrize("M", [16, 33, 48, 144])
@pytest.mark.parametrize("N,K", [(200, 1024), (1536, 1536), (384, 8960)])
def test_tc_quantised_weights_match_oracle(kind, M, N, K):
    w = synth.weights_fp16(N * 7 + K + M, N, K)
    x = synth.activations_fp16(M * 5 + K, M, K)
    wd, sd, w64 = _quant_variant(kind, w)
    y = torch.empty(M, N, dtype=torch.float16, device=dev())
    sq.sq_linear_ex(WKQ[kind], f16_to_dev(x), wd, sd, None, None, sq.SQ_EPI_NONE, y)
    assert sq.sq_check() == 0
    assert_close(dev_to_f64(y), oracle.linear(x.astype(np.float64), w64), f"{kind} M={M} N={N} K={K}")


@pytest.mark.parametrize("kind", ["int4", "fp8"])
def test_tc_quantised_silu_bias(kind):
    I, K, M = 256, 1536, 48
    w = synth.weights_fp16(51, 2 * I, K)
    x = synth.activations_fp16(52, M, K)
    b = synth.fp16_normal(53, (2 * I,), 0.5)
    wd, sd, w64 = _quant_variant(kind, w)
    y = torch.empty(M, I, dtype=torch.float16, device=dev())
    sq.sq_linear_ex(WKQ[kind], f16_to_dev(x), wd, sd, f16_to_dev(b), None, sq.SQ_EPI_SILU_GATE, y)
    full = oracle.linear(x.astype(np.float64), w64, b.astype(np.float64))
    assert_close(dev_to_f64(y), oracle.silu_gate(full[:, :I], full[:, I:]), kind)


def test_tc_fp8_full_size_qkv_7b_sampled():
    _, N, K = QWEN25_7B.projections()[0]
    M = 48
    wt = synth.weights_fp16_device(61, N, K, dev())
    codes = torch.empty(N, K, dtype=torch.uint8, device=dev())
    scales = torch.empty(N, dtype=torch.float32, device=dev())
    sq.sq_quantize(wt, sq.SQ_FP8_E4M3_ROW, codes, scales)
    xt = synth.activations_fp16_device(62, M, K, dev())
    y = torch.empty(M, N, dtype=torch.float16, device=dev())
    sq.sq_linear_fp8(xt, codes, scales, None, y)
    cols = np.unique(np.concatenate([[0, N - 1], np.random.default_rng(7).integers(0, N, 62)]))
    w_rows = bits16(wt[torch.from_numpy(cols).to(dev())]).view(np.float16)
    c, s = oracle.quantize_fp8(w_rows.view(np.uint16))
    x64 = bits16(xt).view(np.float16).astype(np.float64)
    assert_close(dev_to_f64(y)[:, cols], oracle.linear(x64, oracle.dequant_fp8(c, s)), "fp8 7B qkv M=48")


# Below 16 rows the tensor-core path takes the formats and shapes where it
# is faster than the CUDA-core GEMV; rows past M are zero-filled tile rows.
SMALL_M_TC = [
    ("fp16", 3, 384, 8960, sq.SQ_EPI_NONE),      # long rows
    ("fp16", 5, 200, 8192, sq.SQ_EPI_NONE),
    ("fp16", 7, 65600, 2048, sq.SQ_EPI_NONE),    # wide output
    ("fp16", 5, 2816, 3072, sq.SQ_EPI_SILU_GATE),
    ("fp16", 8, 200, 1000, sq.SQ_EPI_NONE),
    ("fp16", 9, 1536, 1536, sq.SQ_EPI_NONE),
    ("fp16", 15, 300, 640, sq.SQ_EPI_NONE),
    ("fp8", 9, 200, 1024, sq.SQ_EPI_NONE),
    ("fp8", 9, 384, 8960, sq.SQ_EPI_NONE),
    ("fp8", 12, 256, 1536, sq.SQ_EPI_SILU_GATE),
    ("int4", 9, 1024, 8192, sq.SQ_EPI_NONE),
    ("int4", 13, 2048, 4096, sq.SQ_EPI_NONE),
]


@pytest.mark.parametrize("kind,M,N,K,epi", SMALL_M_TC)
def test_tc_small_m_matches_oracle(kind, M, N, K, epi):
    wk = {"fp16": sq.SQ_W_FP16, "int4": sq.SQ_W_INT4, "fp8": sq.SQ_W_FP8}[kind]
    assert sq.sq_linear_path(wk, M, N, K, epi) == 1
    silu = epi == sq.SQ_EPI_SILU_GATE
    rows = 2 * N if silu else N
    w = synth.weights_fp16(rows + 3 * K + M, rows, K)
    x = synth.activations_fp16(7 * M + K, M, K)
    if kind == "fp16":
        wd, sd, w64 = f16_to_dev(w), None, w.astype(np.float64)
    else:
        wd, sd, w64 = _quant_variant(kind, w)
    y = torch.empty(M, N, dtype=torch.float16, device=dev())
    sq.sq_linear_ex(wk, f16_to_dev(x), wd, sd, None, None, epi, y)
    assert sq.sq_check() == 0
    full = oracle.linear(x.astype(np.float64), w64)
    ref = oracle.silu_gate(full[:, :N], full[:, N:]) if silu else full
    assert_close(dev_to_f64(y), ref, f"{kind} M={M} N={N} K={K} epi={epi}")


def test_engine_choice_small_rows():
    # few rows and small matrices stay on the CUDA-core GEMV; one INT4 row
    # over many 16-row tiles takes the register-operand tensor-core path
    assert sq.sq_linear_path(sq.SQ_W_INT4, 1, 151936, 1536, sq.SQ_EPI_NONE) == 2
    assert sq.sq_linear_path(sq.SQ_W_INT4, 1, 8960, 1536, sq.SQ_EPI_SILU_GATE) == 2
    assert sq.sq_linear_path(sq.SQ_W_INT4, 1, 2048, 1536, sq.SQ_EPI_NONE) == 0
    assert sq.sq_linear_path(sq.SQ_W_FP8, 1, 151936, 1536, sq.SQ_EPI_NONE) == 0
    assert sq.sq_linear_path(sq.SQ_W_FP16, 5, 2048, 1536, sq.SQ_EPI_NONE) == 0
    assert sq.sq_linear_path(sq.SQ_W_FP16, 5, 151936, 1536, sq.SQ_EPI_NONE) == 0
    # two to eight INT4 / FP8 rows: the shared-memory ring engine
    assert sq.sq_linear_path(sq.SQ_W_FP8, 5, 17920, 1536, sq.SQ_EPI_NONE) == 3
    assert sq.sq_linear_path(sq.SQ_W_INT4, 8, 2048, 1536, sq.SQ_EPI_NONE) == 3
    assert sq.sq_linear_path(sq.SQ_W_INT4, 8, 5120, 13824, sq.SQ_EPI_NONE) == 1  # 8 rows x 13824: no room
    # from 16 rows on: tensor cores
    assert sq.sq_linear_path(sq.SQ_W_INT4, 16, 2048, 1536, sq.SQ_EPI_NONE) == 1
    assert sq.sq_linear_path(sq.SQ_W_FP16, 16, 128, 64, sq.SQ_EPI_NONE) == 1
    # sizes sq_linear_ex rejects
    assert sq.sq_linear_path(sq.SQ_W_INT4, 1, 256, 100, sq.SQ_EPI_NONE) == -1
    assert sq.sq_linear_path(sq.SQ_W_FP16, 0, 256, 256, sq.SQ_EPI_NONE) == -1
    assert sq.sq_linear_path(sq.SQ_W_FP16, 257, 256, 256, sq.SQ_EPI_NONE) == -1


@pytest.mark.parametrize("kind", ["fp16", "int4", "fp8"])
def test_tc_silu_largest_m(kind):
    # M = 256 with the fused gate: the split-K partial tile would not fit in
    # shared memory, so K stays unsplit
    I, K, M = 320, 1536, 256
    w = synth.weights_fp16(71, 2 * I, K)
    x = synth.activations_fp16(72, M, K)
    if kind == "fp16":
        wd, sd, w64 = f16_to_dev(w), None, w.astype(np.float64)
    else:
        wd, sd, w64 = _quant_variant(kind, w)
    wk = {"fp16": sq.SQ_W_FP16, "int4": sq.SQ_W_INT4, "fp8": sq.SQ_W_FP8}[kind]
    y = torch.empty(M, I, dtype=torch.float16, device=dev())
    sq.sq_linear_ex(wk, f16_to_dev(x), wd, sd, None, None, sq.SQ_EPI_SILU_GATE, y)
    assert sq.sq_check() == 0
    full = oracle.linear(x.astype(np.float64), w64)
    assert_close(dev_to_f64(y), oracle.silu_gate(full[:, :I], full[:, I:]), f"{kind} silu M=256")


@pytest.mark.parametrize("M,N,K,epi", [
    (16, 8192, 5120, sq.SQ_EPI_NONE),         # 21.5 MB of INT4: two CTAs per SM, split 4
    (8, 5120, 13824, sq.SQ_EPI_NONE),         # the 14B down shape: split 8
    (16, 2 * 6912, 5120, sq.SQ_EPI_SILU_GATE),  # a fused gate/up of 36 MB: split 2
])
def test_tc_int4_large_matrices_sampled(M, N, K, epi):
    # INT4 matrices of 20 MB and more at few rows take their own split rule;
    # checked on sampled output columns (the oracle dequantises those rows)
    w = synth.weights_fp16(N + K + M, N, K)
    x = synth.activations_fp16(M + 3, M, K)
    c, s = oracle.quantize_int4(w.view(np.uint16))
    y = torch.empty(M, N // 2 if epi == sq.SQ_EPI_SILU_GATE else N, dtype=torch.float16, device=dev())
    assert sq.sq_linear_path(sq.SQ_W_INT4, M, y.shape[1], K, epi) == 1
    sq.sq_linear_ex(sq.SQ_W_INT4, f16_to_dev(x), torch.from_numpy(c).to(dev()), f16_to_dev(s.view(np.float16)),
                    None, None, epi, y)
    assert sq.sq_check() == 0
    ncol = y.shape[1]
    cols = np.unique(np.concatenate([[0, ncol - 1], np.random.default_rng(M).integers(0, ncol, 62)]))
    rows = cols if epi != sq.SQ_EPI_SILU_GATE else np.concatenate([cols, cols + ncol])
    w64 = oracle.dequant_int4(c[rows], s[rows], K)
    ref = oracle.linear(x.astype(np.float64), w64)
    if epi == sq.SQ_EPI_SILU_GATE:
        ref = oracle.silu_gate(ref[:, :len(cols)], ref[:, len(cols):])
    assert_close(dev_to_f64(y)[:, cols], ref, f"int4 M={M} N={N} K={K}")
