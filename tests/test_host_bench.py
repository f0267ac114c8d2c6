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
