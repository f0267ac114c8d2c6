"""GB300-native (sm_103a) SpecQuant draft/verify hot path.

A thin ctypes binding over ``libspecquant.so`` (the C ABI declared in
``include/specquant.h``).  Functions keep the C names and only marshal
arguments: torch tensors supply device memory (``data_ptr()``) and sizes,
``torch.cuda`` supplies the stream.  Every step of the path runs in the
library's CUDA kernels; there is no CPU fallback, and importing a function
fails loudly when the library has not been built.

Paper: "SpecQuant -- Speculative Decoding with Multi-Parent Quantization for
Adaptive LLM Inference" (Sec. III-A variants, Sec. III-D pipeline).
"""
from __future__ import annotations

import ctypes
import os

import torch

from ._build import LIB as LIB_PATH
from ._build import build

__all__ = [
    "SQError", "build", "load", "LIB_PATH",
    "SQ_INT4_G128", "SQ_FP8_E4M3_ROW", "SQ_ACCEPT_SAMPLE", "SQ_ACCEPT_GREEDY",
    "SQ_EPI_NONE", "SQ_EPI_SILU_GATE", "SQ_EPI_RESIDUAL", "SQ_W_FP16", "SQ_W_INT4", "SQ_W_FP8",
    "sq_quantized_bytes", "sq_quantize", "sq_linear_w4a16", "sq_linear_fp8", "sq_verify",
    "sq_linear_ex", "sq_accept_workspace_bytes", "sq_accept", "sq_sample", "sq_check",
    "sq_version", "sq_accept_noalloc", "sq_linear_path", "sq_linear_chain", "SqLinearOp",
    "sq_selftest_wait",
    "sq_accept_logits_workspace_bytes", "sq_accept_logits", "sq_sample_logits",
    "sq_softmax_workspace_bytes", "sq_softmax", "sq_rmsnorm", "sq_kv_append",
    "sq_attention_workspace_bytes", "sq_attention", "sq_kv_rollback", "sq_embed",
    "sq_attention_append", "sq_linear_norm", "sq_spec_commit", "sq_spec_drafts",
    "EXPORTED_SYMBOLS",
]

SQ_OK = 0
SQ_INT4_G128, SQ_FP8_E4M3_ROW = 1, 2
SQ_ACCEPT_SAMPLE, SQ_ACCEPT_GREEDY = 0, 1
SQ_EPI_NONE, SQ_EPI_SILU_GATE, SQ_EPI_RESIDUAL = 0, 1, 2
SQ_W_FP16, SQ_W_INT4, SQ_W_FP8 = 0, 1, 2
SQ_DEV_NONFINITE_WEIGHT, SQ_DEV_BAD_DRAFT_TOKEN, SQ_DEV_NO_MASS, SQ_DEV_BAD_UNIFORM = 1, 2, 4, 8
SQ_DEV_TIMEOUT, SQ_DEV_NONFINITE_LOGIT, SQ_DEV_BAD_POSITION, SQ_DEV_BAD_TOKEN_ID = 0x10, 0x20, 0x40, 0x80

_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_INT = ctypes.c_int
_SIZE = ctypes.c_size_t
_SIGS = {
    "sq_last_error": (ctypes.c_char_p, []),
    "sq_status_string": (ctypes.c_char_p, [_INT]),
    "sq_version": (_INT, []),
    "sq_check": (_INT, [_P, ctypes.POINTER(ctypes.c_uint32)]),
    "sq_quantized_bytes": (_SIZE, [_INT, _I64, _I64, ctypes.POINTER(_SIZE)]),
    "sq_quantize": (_INT, [_P, _I64, _I64, _INT, _P, _P, _P]),
    "sq_linear_w4a16": (_INT, [_P, _P, _P, _P, _P, _INT, _I64, _I64, _P]),
    "sq_linear_fp8": (_INT, [_P, _P, _P, _P, _P, _INT, _I64, _I64, _P]),
    "sq_verify": (_INT, [_P, _P, _P, _P, _INT, _I64, _I64, _P]),
    "sq_linear_ex": (_INT, [_INT, _P, _P, _P, _P, _P, _INT, _P, _INT, _I64, _I64, _P]),
    "sq_linear_norm": (_INT, [_INT, _P, _P, ctypes.c_float, _P, _P, _P, _P, _P, _INT, _P, _INT, _I64,
                              _I64, _P]),
    "sq_accept_workspace_bytes": (_SIZE, [_INT, _INT, _I64]),
    "sq_accept": (_INT, [_P, _P, _P, _P, _INT, _INT, _I64, _INT, _P, _P, _P, _SIZE, _P]),
    "sq_sample": (_INT, [_P, _P, _INT, _I64, _P, _P, _SIZE, _P]),
    "sq_accept_noalloc": (_INT, [_P, _P, _P, _P, _INT, _INT, _I64, _INT, _P, _P, _P]),
    "sq_linear_path": (_INT, [_INT, _INT, _I64, _I64, _INT]),
    "sq_linear_chain": (_INT, [_P, _INT, _P]),
    "sq_selftest_wait": (_INT, [_INT, ctypes.c_uint64, _P]),
    "sq_accept_logits_workspace_bytes": (_SIZE, [_INT, _INT, _I64]),
    "sq_accept_logits": (_INT, [_P, _P, _P, _P, _INT, _INT, _I64, ctypes.c_float, _INT, _P, _P, _P,
                                _SIZE, _P]),
    "sq_sample_logits": (_INT, [_P, _P, _INT, _I64, ctypes.c_float, _P, _P, _SIZE, _P]),
    "sq_softmax_workspace_bytes": (_SIZE, [_I64, _I64]),
    "sq_softmax": (_INT, [_P, _I64, _I64, ctypes.c_float, _P, _P, _SIZE, _P]),
    "sq_rmsnorm": (_INT, [_P, _P, _INT, _I64, ctypes.c_float, _P, _P]),
    "sq_kv_append": (_INT, [_P, _INT, _INT, _INT, _INT, _INT, _P, ctypes.c_float, _P, _P, _I64, _P]),
    "sq_attention_workspace_bytes": (_SIZE, [_INT, _INT, _INT, _INT, _INT, _I64]),
    "sq_attention": (_INT, [_P, _INT, _INT, _INT, _INT, _INT, _P, ctypes.c_float, _P, _P, _I64, _P, _P,
                            _SIZE, _P]),
    "sq_kv_rollback": (_INT, [_P, _P, _INT, _INT, _P, _P]),
    "sq_embed": (_INT, [_P, _INT, _I64, _P, _I64, _I64, _P, _P]),
    "sq_attention_append": (_INT, [_P, _INT, _INT, _INT, _INT, _INT, _P, ctypes.c_float, _P, _P, _I64, _P,
                                   _P, _SIZE, _P]),
    "sq_spec_commit": (_INT, [_P, _P, _INT, _INT, _INT, _P, _INT, _P, _P, _P, _P]),
    "sq_spec_drafts": (_INT, [_P, _P, _INT, _INT, _P, _P, _P]),
}
EXPORTED_SYMBOLS = tuple(_SIGS)

_lib = None


class SQError(RuntimeError):
    """A call into libspecquant returned an error status."""

    def __init__(self, fn: str, status: int, msg: str):
        super().__init__(f"{fn}: {msg} (status {status})")
        self.status = status


def load(path: str | None = None) -> ctypes.CDLL:
    """Load libspecquant.so (built by ``build()``); raises if it is missing."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise ImportError(f"{p} is not built; run paper_2609_21704_gb300.build() (needs nvcc)")
    lib = ctypes.CDLL(p)
    for name, (res, args) in _SIGS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


def _check(fn: str, status: int) -> None:
    if status != SQ_OK:
        lib = load()
        raise SQError(fn, status, lib.sq_last_error().decode(errors="replace"))


def _ptr(t):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError("expected a torch.Tensor")
    if not t.is_cuda:
        raise ValueError("tensor must live on a CUDA device")
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def sq_version() -> int:
    return load().sq_version()


def sq_linear_path(wkind: int, M: int, N: int, K: int, epi: int = SQ_EPI_NONE) -> int:
    """1: tcgen05 tensor-core tiles, 0: CUDA-core GEMV, 2: one INT4 row with
    its products on the tensor cores' register-operand path, 3: one row
    through the shared-memory ring engine, -1: sizes sq_linear_ex rejects."""
    return load().sq_linear_path(wkind, M, N, K, epi)


def sq_quantized_bytes(kind: int, N: int, K: int):
    sb = _SIZE(0)
    cb = load().sq_quantized_bytes(kind, N, K, ctypes.byref(sb))
    return int(cb), int(sb.value)


def sq_quantize(w16, kind, codes, scales, stream=None) -> None:
    N, K = w16.shape
    _check("sq_quantize", load().sq_quantize(_ptr(w16), N, K, kind, _ptr(codes), _ptr(scales),
                                             _stream(stream)))


def sq_linear_ex(wkind, x, w, scales, bias, residual, epi, y, stream=None) -> None:
    M, K = x.shape
    N = y.shape[1]
    _check("sq_linear_ex", load().sq_linear_ex(wkind, _ptr(x), _ptr(w), _ptr(scales), _ptr(bias),
                                               _ptr(residual), epi, _ptr(y), M, N, K,
                                               _stream(stream)))


def sq_linear_norm(wkind, x, gamma, eps, xn, w, scales, bias, residual, epi, y, stream=None) -> None:
    """y = linear(rmsnorm(x) * gamma); xn fp16 [M, K] scratch for the
    normalised rows (written only where the engine needs them in memory)."""
    M, K = x.shape
    N = y.shape[1]
    _check("sq_linear_norm", load().sq_linear_norm(wkind, _ptr(x), _ptr(gamma), float(eps), _ptr(xn), _ptr(w),
                                                   _ptr(scales), _ptr(bias), _ptr(residual), epi, _ptr(y),
                                                   M, N, K, _stream(stream)))


class SqLinearOp(ctypes.Structure):
    """Mirror of the C struct sq_linear_op."""
    _fields_ = [("wkind", ctypes.c_int), ("epi", ctypes.c_int), ("M", ctypes.c_int),
                ("reserved", ctypes.c_int), ("N", ctypes.c_int64), ("K", ctypes.c_int64),
                ("x", _P), ("w", _P), ("scales", _P), ("bias", _P), ("residual", _P), ("y", _P)]


def sq_linear_chain(ops, stream=None) -> None:
    """ops: sequence of (wkind, x, w, scales, bias, residual, epi, y) with the
    same meaning as sq_linear_ex's arguments; run in order (one C call)."""
    arr = _op_array(ops)
    _check("sq_linear_chain", load().sq_linear_chain(ctypes.cast(arr, _P), len(ops), _stream(stream)))


def _op_array(ops):
    arr = (SqLinearOp * max(1, len(ops)))()
    for i, (wkind, x, w, scales, bias, residual, epi, y) in enumerate(ops):
        M, K = x.shape
        arr[i] = SqLinearOp(wkind, epi, M, 0, y.shape[1], K, _ptr(x), _ptr(w), _ptr(scales),
                            _ptr(bias), _ptr(residual), _ptr(y))
    return arr


def sq_selftest_wait(which: int, limit: int, stream=None) -> None:
    """Make one bounded device wait run out (0: poll-bounded, `limit` polls;
    1: time-bounded, `limit` ns); the next sq_check reports SQ_DEV_TIMEOUT."""
    _check("sq_selftest_wait", load().sq_selftest_wait(which, limit, _stream(stream)))


def sq_linear_w4a16(x, codes, scales, bias, y, stream=None) -> None:
    M, K = x.shape
    N = y.shape[1]
    _check("sq_linear_w4a16", load().sq_linear_w4a16(_ptr(x), _ptr(codes), _ptr(scales), _ptr(bias),
                                                     _ptr(y), M, N, K, _stream(stream)))


def sq_linear_fp8(x, codes, scales, bias, y, stream=None) -> None:
    M, K = x.shape
    N = y.shape[1]
    _check("sq_linear_fp8", load().sq_linear_fp8(_ptr(x), _ptr(codes), _ptr(scales), _ptr(bias),
                                                 _ptr(y), M, N, K, _stream(stream)))


def sq_verify(x, w16, bias, y, stream=None) -> None:
    M, K = x.shape
    N = y.shape[1]
    _check("sq_verify", load().sq_verify(_ptr(x), _ptr(w16), _ptr(bias), _ptr(y), M, N, K,
                                         _stream(stream)))


def sq_accept_logits_workspace_bytes(B: int, K: int, V: int) -> int:
    return int(load().sq_accept_logits_workspace_bytes(B, K, V))


def sq_accept_logits(zp, zq, draft, u, temperature, mode, n_accepted, tokens, workspace,
                     stream=None) -> None:
    """zp fp16 [B,K+1,V] target logits, zq fp16 [K,B,V] draft logits (or None)."""
    B, K1, V = zp.shape
    _check("sq_accept_logits", load().sq_accept_logits(
        _ptr(zp), _ptr(zq), _ptr(draft), _ptr(u), B, K1 - 1, V, float(temperature), mode,
        _ptr(n_accepted), _ptr(tokens), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def sq_sample_logits(z, u, temperature, tokens, workspace, stream=None) -> None:
    """token[b] ~ softmax(z[b] / T); z fp16 [B, V]."""
    B, V = z.shape
    _check("sq_sample_logits", load().sq_sample_logits(
        _ptr(z), _ptr(u), B, V, float(temperature), _ptr(tokens), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def sq_softmax_workspace_bytes(R: int, V: int) -> int:
    return int(load().sq_softmax_workspace_bytes(R, V))


def sq_softmax(z, temperature, p, workspace, stream=None) -> None:
    """p fp32 [R, V] = softmax(z / T) row by row; z fp16 [R, V]."""
    R, V = z.shape
    _check("sq_softmax", load().sq_softmax(_ptr(z), R, V, float(temperature), _ptr(p), _ptr(workspace),
                                           workspace.numel() * workspace.element_size(),
                                           _stream(stream)))


def sq_rmsnorm(x, gamma, eps, y, stream=None) -> None:
    M, H = x.shape
    _check("sq_rmsnorm", load().sq_rmsnorm(_ptr(x), _ptr(gamma), M, H, float(eps), _ptr(y),
                                           _stream(stream)))


def sq_kv_append(qkv, B, T, Hq, Hkv, pos0, theta, k_cache, v_cache, stream=None) -> None:
    """qkv fp16 [B*T, (Hq+2Hkv)*128]; caches fp16 [B, Hkv, max_ctx, 128]."""
    _check("sq_kv_append", load().sq_kv_append(_ptr(qkv), B, T, Hq, Hkv, 128, _ptr(pos0), float(theta),
                                               _ptr(k_cache), _ptr(v_cache), k_cache.shape[2],
                                               _stream(stream)))


def sq_attention_workspace_bytes(B, T, Hq, Hkv, max_ctx) -> int:
    return int(load().sq_attention_workspace_bytes(B, T, Hq, Hkv, 128, max_ctx))


def sq_attention(qkv, B, T, Hq, Hkv, pos0, theta, k_cache, v_cache, out, workspace,
                 stream=None) -> None:
    """out fp16 [B*T, Hq*128] = causal GQA attention of the new tokens over the caches."""
    _check("sq_attention", load().sq_attention(
        _ptr(qkv), B, T, Hq, Hkv, 128, _ptr(pos0), float(theta), _ptr(k_cache), _ptr(v_cache),
        k_cache.shape[2], _ptr(out), _ptr(workspace), workspace.numel() * workspace.element_size(),
        _stream(stream)))


def sq_attention_append(qkv, B, T, Hq, Hkv, pos0, theta, k_cache, v_cache, out, workspace,
                        stream=None) -> None:
    """sq_kv_append + sq_attention in one launch (the caches are written)."""
    _check("sq_attention_append", load().sq_attention_append(
        _ptr(qkv), B, T, Hq, Hkv, 128, _ptr(pos0), float(theta), _ptr(k_cache), _ptr(v_cache),
        k_cache.shape[2], _ptr(out), _ptr(workspace), workspace.numel() * workspace.element_size(),
        _stream(stream)))


def sq_kv_rollback(base, n_accepted, limit, length, stream=None) -> None:
    _check("sq_kv_rollback", load().sq_kv_rollback(_ptr(base), _ptr(n_accepted), base.numel(), limit,
                                                   _ptr(length), _stream(stream)))


def sq_embed(ids, table, out, stream=None, ids_stride: int = 1, M: int | None = None) -> None:
    """out[m] = table[ids[m * ids_stride]] for m < M (default ids.numel());
    ids int32, table fp16 [V, H], out fp16 [M, H]."""
    V, H = table.shape
    if M is None:
        M = ids.numel()
    _check("sq_embed", load().sq_embed(_ptr(ids), M, ids_stride, _ptr(table), V, H, _ptr(out),
                                       _stream(stream)))


def sq_spec_commit(n_accepted, tokens, hist, length, pos, last2, K: int, stream=None) -> None:
    """Append each sequence's n_accepted[b] + 1 committed tokens (tokens int32
    [B, ldt]; n_accepted None = one token) to hist int32 [B, cap] and
    length [B]; write the next cycle's positions pos int32 [K + 1, B] and
    the last two tokens last2 int32 [B, 2]."""
    B, cap = hist.shape
    ldt = tokens.shape[-1] if tokens.dim() > 1 else 1
    _check("sq_spec_commit", load().sq_spec_commit(_ptr(n_accepted), _ptr(tokens), ldt, B, K, _ptr(hist),
                                                   cap, _ptr(length), _ptr(pos), _ptr(last2),
                                                   _stream(stream)))


def sq_spec_drafts(samples, last2, verify_tokens, draft, stream=None) -> None:
    """verify_tokens [B, K+1] = (last token, drafts), draft [B, K] =
    samples^T from the draft steps' tokens samples int32 [K, B]."""
    B, K1 = verify_tokens.shape
    _check("sq_spec_drafts", load().sq_spec_drafts(_ptr(samples), _ptr(last2), B, K1 - 1,
                                                   _ptr(verify_tokens), _ptr(draft), _stream(stream)))


def sq_accept_workspace_bytes(B: int, K: int, V: int) -> int:
    return int(load().sq_accept_workspace_bytes(B, K, V))


def sq_accept(p, q, draft, u, mode, n_accepted, tokens, workspace, stream=None) -> None:
    B, K1, V = p.shape
    _check("sq_accept", load().sq_accept(_ptr(p), _ptr(q), _ptr(draft), _ptr(u), B, K1 - 1, V, mode,
                                         _ptr(n_accepted), _ptr(tokens), _ptr(workspace),
                                         workspace.numel() * workspace.element_size(),
                                         _stream(stream)))


def sq_accept_noalloc(p, q, draft, u, mode, n_accepted, tokens, stream=None) -> None:
    """sq_accept without a workspace, for callers that cannot allocate
    device memory: the library's static 1 MiB scratch is used instead."""
    B, K1, V = p.shape
    _check("sq_accept_noalloc", load().sq_accept_noalloc(_ptr(p), _ptr(q), _ptr(draft), _ptr(u), B,
                                                         K1 - 1, V, mode, _ptr(n_accepted),
                                                         _ptr(tokens), _stream(stream)))


def sq_sample(probs, u, tokens, workspace, stream=None) -> None:
    B, V = probs.shape
    _check("sq_sample", load().sq_sample(_ptr(probs), _ptr(u), B, V, _ptr(tokens), _ptr(workspace),
                                         workspace.numel() * workspace.element_size(),
                                         _stream(stream)))


def sq_check(stream=None) -> int:
    """Synchronise the stream; return the device status bits (0 when clean)."""
    bits = ctypes.c_uint32(0)
    st = load().sq_check(_stream(stream), ctypes.byref(bits))
    if st not in (SQ_OK, 7):
        _check("sq_check", st)
    return int(bits.value)
