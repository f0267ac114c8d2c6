"""The C-ABI library: it loads, exports every function include/specquant.h
declares, and its host-side logic (sizes, validation, status strings)
behaves as documented.  No call here reaches a kernel, so these run
without a GPU."""
import ctypes
import os
import re

import pytest

import paper_2609_21704_gb300 as sq

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "specquant.h")


@pytest.fixture(scope="module")
def lib():
    sq.build()
    return sq.load()


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(sq_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = _declared_functions()
    for want in ("sq_quantize", "sq_linear_w4a16", "sq_linear_fp8", "sq_verify", "sq_accept",
                 "sq_sample", "sq_check", "sq_last_error"):
        assert want in names


def test_every_declared_symbol_is_exported(lib):
    for name in _declared_functions():
        assert hasattr(lib, name), name
    assert set(_declared_functions()) <= set(sq.EXPORTED_SYMBOLS) | {"sq_last_error"}


def test_library_is_built_for_sm_103a_only():
    """The build asks nvcc for exactly one target, sm_103a machine code, and
    no PTX (code=sm_103a, not compute_103a): a device that is not sm_103a
    cannot run the library at all, so a kernel that runs is the sm_103a one
    (tests/test_gpu_quantize.py::test_runs_on_sm_103a checks the device)."""
    from paper_2609_21704_gb300 import _build

    assert _build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]
    assert not any("gencode" in f or "arch=" in f for f in _build.NVCC_FLAGS)


def test_version_and_status_strings(lib):
    assert sq.sq_version() >= 100
    assert lib.sq_status_string(0) == b"SQ_OK"
    assert lib.sq_status_string(5) == b"SQ_ERR_WORKSPACE"
    assert lib.sq_status_string(99) == b"SQ_STATUS_UNKNOWN"


def test_quantized_bytes():
    assert sq.sq_quantized_bytes(sq.SQ_INT4_G128, 4864, 896) == (4864 * 448, 4864 * 7 * 2)
    assert sq.sq_quantized_bytes(sq.SQ_FP8_E4M3_ROW, 10, 32) == (320, 40)
    assert sq.sq_quantized_bytes(sq.SQ_INT4_G128, 4, 100) == (0, 0)
    assert sq.sq_quantized_bytes(sq.SQ_FP8_E4M3_ROW, 4, 24) == (0, 0)
    assert sq.sq_quantized_bytes(7, 4, 128) == (0, 0)


def test_accept_workspace_bytes():
    b = sq.sq_accept_workspace_bytes(8, 5, 152064)
    chunks = (152064 + 2047) // 2048
    assert b >= 8 * chunks * 6 * 8 + 8 * 4
    assert sq.sq_accept_workspace_bytes(1, 17, 100) == 0
    assert sq.sq_accept_workspace_bytes(1, 2, 1 << 20) == 0


def _err(lib):
    return lib.sq_last_error().decode()


def test_validation_rejects_before_launch(lib):
    P = ctypes.c_void_p
    fake = P(4096)  # never dereferenced: validation fails first
    # shape errors
    assert lib.sq_linear_w4a16(fake, fake, fake, None, fake, 0, 16, 128, None) == 2
    assert "M" in _err(lib)
    assert lib.sq_linear_w4a16(fake, fake, fake, None, fake, 1, 16, 100, None) == 2
    assert lib.sq_linear_fp8(fake, fake, fake, None, fake, 1, 16, 24, None) == 2
    assert lib.sq_verify(fake, fake, None, fake, 300, 16, 64, None) == 2
    # null pointers
    assert lib.sq_verify(None, fake, None, fake, 1, 16, 64, None) == 1
    assert lib.sq_linear_w4a16(fake, fake, None, None, fake, 1, 16, 128, None) == 1
    # alignment
    assert lib.sq_verify(P(4098), fake, None, fake, 1, 16, 64, None) == 3
    # unknown enums
    assert lib.sq_linear_ex(9, fake, fake, None, None, None, 0, fake, 1, 16, 64, None) == 1
    assert lib.sq_linear_ex(0, fake, fake, None, None, None, 9, fake, 1, 16, 64, None) == 1
    assert lib.sq_linear_ex(0, fake, fake, None, None, None, 2, fake, 1, 16, 64, None) == 1
    assert lib.sq_quantize(fake, 4, 128, 3, fake, fake, None) == 1
    assert lib.sq_quantize(fake, 4, 100, 1, fake, fake, None) == 2
    assert lib.sq_quantize(fake, 0, 128, 1, None, None, None) == 0  # empty: nothing to do


def test_accept_validation(lib):
    P = ctypes.c_void_p
    fake = P(4096)
    ws_need = sq.sq_accept_workspace_bytes(2, 3, 1000)
    # workspace too small
    assert lib.sq_accept(fake, fake, fake, fake, 2, 3, 1000, 0, fake, fake, fake, ws_need - 1, None) == 5
    # missing q in sampling mode
    assert lib.sq_accept(fake, None, fake, fake, 2, 3, 1000, 0, fake, fake, fake, ws_need, None) == 1
    # K too large, V too large, bad mode
    assert lib.sq_accept(fake, fake, fake, fake, 2, 17, 1000, 0, fake, fake, fake, 1 << 20, None) == 2
    assert lib.sq_accept(fake, fake, fake, fake, 2, 3, 1 << 20, 0, fake, fake, fake, 1 << 30, None) == 2
    assert lib.sq_accept(fake, fake, fake, fake, 2, 3, 1000, 5, fake, fake, fake, ws_need, None) == 1
    # empty batch is a no-op
    assert lib.sq_accept(None, None, None, None, 0, 3, 1000, 0, None, None, None, 0, None) == 0
    # workspace misaligned
    assert lib.sq_sample(fake, fake, 2, 1000, fake, P(4100), 1 << 20, None) == 3


def test_binding_fails_loudly_without_the_library(tmp_path):
    with pytest.raises(ImportError):
        sq.load(str(tmp_path / "missing.so"))


def test_single_row_engine_choice(lib):
    """sq_linear_path is host logic: one activation row takes the shared-
    memory ring (3) for the large matrices where it measured faster (INT4
    fused gate/up of >= 64 Mi weights, FP16 fused gate/up of >= 16 Mi and
    lm_head rows, FP8 lm_head of >= 400 Mi weights), two to eight INT4 or
    FP8 rows take it whenever their activations fit; otherwise one INT4 row
    over at least 192 16-row output tiles takes the register-operand tensor
    path (2) and other few-row calls the streaming CUDA-core GEMV (0).  (The
    tcgen05 path (1) needs a device to encode its tensor maps: checked in
    tests/test_gpu_tc.py.)"""
    W4, W8, W16 = sq.SQ_W_INT4, sq.SQ_W_FP8, sq.SQ_W_FP16
    NONE, SILU, RES = sq.SQ_EPI_NONE, sq.SQ_EPI_SILU_GATE, sq.SQ_EPI_RESIDUAL
    assert sq.sq_linear_path(W4, 1, 8960, 1536, SILU) == 2      # 1.5B fused gate/up (27.5 Mi)
    assert sq.sq_linear_path(W4, 1, 151936, 1536, NONE) == 2    # 1.5B lm_head
    assert sq.sq_linear_path(W4, 1, 18944, 3584, SILU) == 3     # 7B fused gate/up (136 Mi)
    assert sq.sq_linear_path(W4, 1, 13824, 5120, SILU) == 3     # 14B fused gate/up
    assert sq.sq_linear_path(W4, 1, 152064, 5120, NONE) == 2    # 14B lm_head
    assert sq.sq_linear_path(W4, 1, 2048, 1536, NONE) == 0      # 1.5B q/k/v
    assert sq.sq_linear_path(W4, 1, 1536, 1536, RES) == 0       # 1.5B o
    assert sq.sq_linear_path(W4, 1, 1536, 8960, RES) == 0       # 1.5B down
    assert sq.sq_linear_path(W4, 1, 16 * 192, 896, NONE) == 2   # exactly 192 tiles
    assert sq.sq_linear_path(W4, 1, 16 * 192 - 16, 896, NONE) == 0
    assert sq.sq_linear_path(W4, 1, 16 * 191 + 1, 896, NONE) == 2  # ragged 192nd tile
    assert sq.sq_linear_path(W4, 1, 4608, 3584, NONE) == 2      # 7B q/k/v (288 tiles)
    assert sq.sq_linear_path(W4, 1, 3584, 18944, RES) == 2      # 7B down (224 tiles)
    assert sq.sq_linear_path(W4, 1, 32768, 2176, SILU) == 2     # 17 groups: odd, not the ring
    assert sq.sq_linear_path(W4, 2, 151936, 1536, NONE) == 3    # two rows: the ring too
    assert sq.sq_linear_path(W8, 8, 7168, 5120, NONE) == 3      # FP8 draft at batch 8
    assert sq.sq_linear_path(W16, 2, 2048, 1536, NONE) == 0     # FP16 rows: not the ring
    assert sq.sq_linear_path(W4, 9, 2048, 1536, NONE) == 0      # nine rows: not the ring
    assert sq.sq_linear_path(W8, 1, 151936, 1536, NONE) == 0    # 1.5B FP8 lm_head (233 Mi)
    assert sq.sq_linear_path(W8, 1, 152064, 5120, NONE) == 3    # 14B FP8 lm_head (779 Mi)
    assert sq.sq_linear_path(W8, 1, 13824, 5120, SILU) == 0
    assert sq.sq_linear_path(W16, 1, 151936, 1536, NONE) == 3   # FP16 lm_head
    assert sq.sq_linear_path(W16, 1, 8960, 1536, SILU) == 3     # FP16 fused gate/up (27.5 Mi)
    assert sq.sq_linear_path(W16, 1, 4864, 896, SILU) == 0      # 0.5B-shaped (8.7 Mi)
    assert sq.sq_linear_path(W16, 1, 2048, 1536, NONE) == 0
    assert sq.sq_linear_path(W16, 5, 151936, 1536, NONE) == 0   # five rows: not the ring
