"""sq_accept_noalloc: the accept step for callers that cannot allocate
device memory where they run it (a host framework that owns every device
byte through its own pool, or a latency-critical loop where an allocation,
which may synchronise the device, is not acceptable).  Its scratch is the
library's static 1 MiB device array, so the caller passes only inputs and
outputs.

This file is collected last on purpose: a run that stops at the first
failure has already run every other test.  Each check calls the new entry
point through the C ABI twice in a row (different inputs, so the second call
runs on the scratch the first one left behind) and compares it with
sq_accept on a fresh caller workspace; accept results are compared bit for
bit, as in the other accept tests."""
import ctypes

import numpy as np
import pytest
import torch

import paper_2609_21704_gb300 as sq
from paper_2609_21704_gb300 import synth

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda:0")


def _with_workspace(p, q, draft, u, mode):
    B, K1, V = p.shape
    ws = torch.zeros(sq.sq_accept_workspace_bytes(B, K1 - 1, V), dtype=torch.uint8, device="cuda:0")
    n = torch.full((B,), -7, dtype=torch.int32, device="cuda:0")
    tok = torch.full((B, K1), -7, dtype=torch.int32, device="cuda:0")
    sq.sq_accept(p, q, draft, u, mode, n, tok, ws)
    return n, tok


def _no_alloc_via_c_abi(p, q, draft, u, mode):
    lib = sq.load()
    B, K1, V = p.shape
    n = torch.full((B,), -7, dtype=torch.int32, device="cuda:0")
    tok = torch.full((B, K1), -7, dtype=torch.int32, device="cuda:0")
    stream = torch.cuda.current_stream().cuda_stream
    st = lib.sq_accept_noalloc(p.data_ptr(), None if q is None else q.data_ptr(), draft.data_ptr(),
                               u.data_ptr(), B, K1 - 1, V, mode, n.data_ptr(), tok.data_ptr(), stream)
    assert st == 0, lib.sq_last_error()
    return n, tok


@pytest.mark.parametrize("mode", [sq.SQ_ACCEPT_SAMPLE, sq.SQ_ACCEPT_GREEDY])
def test_two_calls_in_a_row_match_sq_accept(mode):
    cases = [(8, 5, 152064, 31), (3, 4, 32000, 32)]  # second call: different B, K, V
    for B, K, V, seed in cases:
        p, q, draft, u = synth.spec_block(seed, B, K, V, draft_noise=0.5)
        if mode == sq.SQ_ACCEPT_GREEDY:
            draft[:, :2] = p[:, :2].argmax(axis=2)  # some agreement
        args = (_dev(p), _dev(q), _dev(draft), _dev(u))
        n_ref, tok_ref = _with_workspace(*args, mode)
        n_got, tok_got = _no_alloc_via_c_abi(*args, mode)
        assert sq.sq_check() == 0
        assert torch.equal(n_got, n_ref)
        assert torch.equal(tok_got, tok_ref)


def test_repeated_identical_calls_agree():
    p, q, draft, u = synth.spec_block(33, 4, 8, 151936, draft_noise=None)
    args = (_dev(p), _dev(q), _dev(draft), _dev(u))
    first = _no_alloc_via_c_abi(*args, sq.SQ_ACCEPT_SAMPLE)
    second = _no_alloc_via_c_abi(*args, sq.SQ_ACCEPT_SAMPLE)
    ref = _with_workspace(*args, sq.SQ_ACCEPT_SAMPLE)
    for a, b in zip(first + second, ref + ref):
        assert torch.equal(a, b)


def test_batches_beyond_the_static_scratch_are_rejected():
    lib = sq.load()
    fake = ctypes.c_void_p(4096)  # never touched: the size check comes first
    too_big = 400  # V = 152064, K = 4 fits at most 349 sequences in 1 MiB
    st = lib.sq_accept_noalloc(fake, fake, fake, fake, too_big, 4, 152064, 0, fake, fake, None)
    assert st == 2
    assert b"static scratch" in lib.sq_last_error()
