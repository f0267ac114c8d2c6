"""Host logic of bench.py's CPU baselines (no GPU): the all-cores oracle run
splits every sample matrix into output-row slices that cover each output
exactly once and together compute what the whole matrix computes."""
import numpy as np
import pytest

import bench
import oracle


def _item(n, k, silu, seed):
    rng = np.random.default_rng(seed)
    w16 = (rng.standard_normal((n, k)) * 0.02).astype(np.float16).view(np.uint16)
    q = oracle.quantize_int4(w16)
    xd = rng.standard_normal((1, k)).astype(np.float16).astype(np.float64)
    xv = rng.standard_normal((5, k)).astype(np.float16).astype(np.float64)
    return (n, k, silu, w16, q, xd, xv)


def _outputs(item):
    n, k, silu, w16, (codes, sc), xd, xv = item
    y = oracle.linear(xd, oracle.dequant_int4(codes, sc, k))
    return oracle.silu_gate(y[:, : n // 2], y[:, n // 2:]) if silu else y


@pytest.mark.parametrize("n,silu", [(40, False), (38, True), (7, False)])
@pytest.mark.parametrize("P", [1, 3, 8])
def test_row_slices_partition_and_reproduce_the_outputs(n, silu, P):
    it = _item(n, 128, silu, n * 10 + P)
    parts = [bench._row_slice(it, w, P) for w in range(P)]
    assert sum(p[0] for p in parts) == n
    # the slices' rows, in order, are the whole matrix's rows, once each
    half = n // 2 if silu else n
    got = np.concatenate([_outputs(p) for p in parts if p[0] > 0], axis=1)
    assert got.shape[1] == half
    np.testing.assert_array_equal(got, _outputs(it))


def test_workload_name_names_the_stack_and_the_cycle():
    """Both arms name their workload with bench.workload_name: the stack,
    its linear weight count, the draft and verify rows of one cycle and the
    vocabulary the accept runs over."""
    from paper_2609_21704_gb300.shapes import QWEN25_14B, QWEN25_7B

    assert bench.workload_name(QWEN25_14B, "int4", 1, 4) == (
        "qwen2.5-14b linear stack (48 layers + lm_head, 13.991B linear weights), INT4 draft "
        "B=1 x K=4 (M=1), FP16 verify M=5, accept V=152064")
    name = bench.workload_name(QWEN25_7B, "fp8", 8, 5)
    assert "FP8 draft B=8 x K=5 (M=8)" in name and "FP16 verify M=48" in name
    assert f"{QWEN25_7B.linear_params() / 1e9:.3f}B" in name
