"""GPU: the failure path of the bounded device waits.

Every wait inside the library's kernels (the tcgen05 tile path's mbarrier
polls, the ring engine's timed mbarrier waits) is bounded; a wait that runs
out sets SQ_DEV_TIMEOUT and the kernel finishes.  sq_selftest_wait makes
one such wait run out on purpose, with nothing else in flight, so this test
needs no fault: it checks that the status bit reaches sq_check, that
sq_check clears it, and that the same stream then runs linear layers and
the accept step correctly."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq
from paper_2609_21704_gb300 import synth

from gpu_util import assert_close, dev, dev_to_f64, f16_to_dev

pytestmark = pytest.mark.gpu


def _linear_still_works(stream, M):
    N, K = 300, 1024
    w = synth.weights_fp16(41, N, K)
    x = synth.activations_fp16(42, M, K)
    y = torch.empty(M, N, dtype=torch.float16, device=dev())
    with torch.cuda.stream(stream):
        sq.sq_linear_ex(sq.SQ_W_FP16, f16_to_dev(x), f16_to_dev(w), None, None, None, sq.SQ_EPI_NONE, y,
                        stream)
    assert sq.sq_check(stream) == 0
    assert_close(dev_to_f64(y), oracle.linear(x.astype(np.float64), w.astype(np.float64)), f"M={M}")


@pytest.mark.parametrize("which,limit", [(0, 1000), (1, 200_000)])
def test_wait_runs_out_and_device_stays_usable(which, limit):
    assert sq.sq_check() == 0
    s = torch.cuda.Stream()
    sq.sq_selftest_wait(which, limit, s)
    assert sq.sq_check(s) == sq.SQ_DEV_TIMEOUT
    assert sq.sq_check(s) == 0  # read and cleared
    # the same stream runs the GEMV, the tensor-core tile path and the accept
    _linear_still_works(s, 1)
    _linear_still_works(s, 32)
    B, K, V = 2, 4, 32000
    p, q, d, u = synth.spec_block(7, B, K, V)
    n = torch.empty(B, dtype=torch.int32, device=dev())
    t = torch.empty(B, K + 1, dtype=torch.int32, device=dev())
    ws = torch.zeros(sq.sq_accept_workspace_bytes(B, K, V), dtype=torch.uint8, device=dev())
    with torch.cuda.stream(s):
        sq.sq_accept(*(torch.from_numpy(a).to(dev()) for a in (p, q, d, u)), sq.SQ_ACCEPT_SAMPLE, n, t, ws, s)
    assert sq.sq_check(s) == 0
    _, on, ot = oracle.accept(p, q, d, u, oracle.ACCEPT_SAMPLE)
    assert np.array_equal(n.cpu().numpy(), on) and np.array_equal(t.cpu().numpy(), ot)


def test_selftest_rejects_bad_arguments():
    for which, limit in ((2, 10), (0, 0), (0, 1 << 25), (1, 0), (1, 2_000_000_000)):
        with pytest.raises(sq.SQError):
            sq.sq_selftest_wait(which, limit)
    assert sq.sq_check() == 0
