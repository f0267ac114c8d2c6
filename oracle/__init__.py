"""CPU oracle for the SpecQuant draft/verify hot path.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The CUDA product
path (``paper_2609_21704_gb300``) never imports it and has no CPU fallback.

The arithmetic lives in plain C (``sq_oracle.c``), compiled with gcc without
fast-math and with ``-ffp-contract=off`` so that x86-64 and AArch64 give the
same bits.  This module only marshals numpy arrays.  Each function names the
passage of the paper it follows; the readings taken where the paper is silent
are stated in ``sq_oracle.c``.

Every function is pinned by ``-m "not gpu"`` tests against something other
than itself: numpy/torch casts, brute-force searches, exact rational
arithmetic and exhaustive enumeration of the accept rule.
"""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess
import tempfile

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SOURCES = ("sq_oracle.c", "sq_enumerate.c")
_HEADER = "sq_oracle.h"
_LIB_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_LIB_DIR, "libsq_oracle.so")

ACCEPT_SAMPLE = 0
ACCEPT_GREEDY = 1
OK, BAD_ARG, BAD_SEQ = 0, 1, 2
GROUP = 128

_lib = None


def _stale() -> bool:
    if not os.path.exists(_LIB_PATH):
        return True
    t = os.path.getmtime(_LIB_PATH)
    return any(os.path.getmtime(os.path.join(_HERE, f)) > t for f in _SOURCES + (_HEADER,))


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/_build/libsq_oracle.so`` with gcc."""
    if not force and not _stale():
        return _LIB_PATH
    os.makedirs(_LIB_DIR, exist_ok=True)
    srcs = [os.path.join(_HERE, f) for f in _SOURCES]
    base = ["gcc", "-O2", "-fPIC", "-shared", "-std=gnu11", "-fno-fast-math",
            "-ffp-contract=off", "-Wall"]
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=_LIB_DIR)
    os.close(fd)
    try:
        r = subprocess.run(base + ["-fopenmp"] + srcs + ["-o", tmp, "-lm"],
                           capture_output=True, text=True)
        if r.returncode != 0:  # no OpenMP runtime: the sweep runs on one thread
            r = subprocess.run(base + srcs + ["-o", tmp, "-lm"], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("oracle build failed:\n" + r.stderr)
        shutil.move(tmp, _LIB_PATH)
    finally:
        if os.path.exists(tmp):
            os.unlink(tmp)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    L = ctypes.CDLL(_LIB_PATH)
    P = ctypes.c_void_p
    I64 = ctypes.c_int64
    sig = {
        "oq_f16_decode": (ctypes.c_double, [ctypes.c_uint16]),
        "oq_f16_encode": (ctypes.c_uint16, [ctypes.c_double]),
        "oq_e4m3_decode": (ctypes.c_double, [ctypes.c_uint8]),
        "oq_e4m3_encode": (ctypes.c_uint8, [ctypes.c_double]),
        "oq_f16_decode_array": (None, [P, I64, P]),
        "oq_f16_encode_array": (None, [P, I64, P]),
        "oq_e4m3_encode_array": (None, [P, I64, P]),
        "oq_quantize_int4": (ctypes.c_int, [P, I64, I64, P, P]),
        "oq_dequant_int4": (ctypes.c_int, [P, P, I64, I64, P]),
        "oq_quantize_fp8": (ctypes.c_int, [P, I64, I64, P, P]),
        "oq_dequant_fp8": (ctypes.c_int, [P, P, I64, I64, P]),
        "oq_linear": (None, [P, P, P, I64, I64, I64, P]),
        "oq_silu_gate": (None, [P, P, I64, P]),
        "oq_fix44": (ctypes.c_uint64, [ctypes.c_float]),
        "oq_scale_floor": (ctypes.c_uint64, [ctypes.c_float, ctypes.c_uint64]),
        "oq_accept": (ctypes.c_int, [P, P, P, P, I64, I64, I64, ctypes.c_int, P, P]),
        "oq_sample": (ctypes.c_int, [P, P, I64, I64, P]),
        "oq_enum_sweep": (ctypes.c_int, [P, P, P, P, I64, I64, ctypes.c_int, ctypes.c_int,
                                         ctypes.c_int, P]),
        "oq_rmsnorm": (None, [P, P, I64, I64, ctypes.c_double, P]),
        "oq_rope": (None, [P, P, I64, I64, I64, ctypes.c_double]),
        "oq_attention": (None, [P, P, P, P, I64, I64, I64, I64, I64, P]),
        "oq_exp_neg": (ctypes.c_float, [ctypes.c_float]),
        "oq_exp_neg_array": (None, [P, I64, P]),
        "oq_softmax_row": (ctypes.c_int, [P, I64, ctypes.c_float, P]),
        "oq_accept_logits": (ctypes.c_int, [P, P, P, P, I64, I64, I64, ctypes.c_float, ctypes.c_int,
                                            P, P]),
        "oq_sample_logits": (ctypes.c_int, [P, P, I64, I64, ctypes.c_float, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def _c(a: np.ndarray, dtype) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=dtype)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


# ---- number formats ----------------------------------------------------------

def f16_decode(bits) -> np.ndarray:
    """binary16 bit patterns -> exact float64 values (IEEE 754)."""
    b = _c(bits, np.uint16)
    out = np.empty(b.shape, np.float64)
    _load().oq_f16_decode_array(_ptr(b), b.size, _ptr(out))
    return out


def f16_encode(x) -> np.ndarray:
    """float64 -> nearest binary16 bit pattern, ties to even."""
    a = _c(x, np.float64)
    out = np.empty(a.shape, np.uint16)
    _load().oq_f16_encode_array(_ptr(a), a.size, _ptr(out))
    return out


def e4m3_decode(codes) -> np.ndarray:
    L = _load()
    c = _c(codes, np.uint8)
    return np.array([L.oq_e4m3_decode(int(v)) for v in c.ravel()], np.float64).reshape(c.shape)


def e4m3_encode(x) -> np.ndarray:
    """float32 -> E4M3 bits, round to nearest even, saturating to +-448."""
    a = _c(x, np.float32)
    out = np.empty(a.shape, np.uint8)
    _load().oq_e4m3_encode_array(_ptr(a), a.size, _ptr(out))
    return out


# ---- Sec. III-A.1 / III-A.2: derive the variants ----------------------------

def quantize_int4(w16_bits):
    """Q4 = f(W16, 4): fp16 bits [N,K] -> (codes u8 [N,K/2], scales fp16 bits [N,K/128])."""
    w = _c(w16_bits, np.uint16)
    N, K = w.shape
    codes = np.zeros((N, K // 2), np.uint8)
    scales = np.zeros((N, max(K // GROUP, 0)), np.uint16)
    st = _load().oq_quantize_int4(_ptr(w), N, K, _ptr(codes), _ptr(scales))
    if st != OK:
        raise ValueError(f"oq_quantize_int4 rejected the input (status {st})")
    return codes, scales


def dequant_int4(codes, scales, K: int) -> np.ndarray:
    c = _c(codes, np.uint8)
    s = _c(scales, np.uint16)
    N = c.shape[0]
    w = np.empty((N, K), np.float64)
    st = _load().oq_dequant_int4(_ptr(c), _ptr(s), N, K, _ptr(w))
    if st != OK:
        raise ValueError(f"oq_dequant_int4 status {st}")
    return w


def quantize_fp8(w16_bits):
    """Q8 = f(W16, 8): fp16 bits [N,K] -> (codes E4M3 u8 [N,K], scales f32 [N])."""
    w = _c(w16_bits, np.uint16)
    N, K = w.shape
    codes = np.zeros((N, K), np.uint8)
    scales = np.zeros((N,), np.float32)
    st = _load().oq_quantize_fp8(_ptr(w), N, K, _ptr(codes), _ptr(scales))
    if st != OK:
        raise ValueError(f"oq_quantize_fp8 rejected the input (status {st})")
    return codes, scales


def dequant_fp8(codes, scales) -> np.ndarray:
    c = _c(codes, np.uint8)
    s = _c(scales, np.float32)
    N, K = c.shape
    w = np.empty((N, K), np.float64)
    _load().oq_dequant_fp8(_ptr(c), _ptr(s), N, K, _ptr(w))
    return w


# ---- Sec. III-D.2 / III-D.3: linear layers ----------------------------------

def linear(x, w, bias=None) -> np.ndarray:
    """y = x w^T (+ bias) in fp64; x [M,K], w [N,K] as float64."""
    xa = _c(x, np.float64)
    wa = _c(w, np.float64)
    ba = None if bias is None else _c(bias, np.float64)
    M, K = xa.shape
    N = wa.shape[0]
    assert wa.shape[1] == K
    y = np.empty((M, N), np.float64)
    _load().oq_linear(_ptr(xa), _ptr(wa), _ptr(ba), M, N, K, _ptr(y))
    return y


def silu_gate(g, u) -> np.ndarray:
    ga = _c(g, np.float64)
    ua = _c(u, np.float64)
    h = np.empty(ga.shape, np.float64)
    _load().oq_silu_gate(_ptr(ga), _ptr(ua), ga.size, _ptr(h))
    return h


# ---- Sec. III-A.3 / III-D.4: accept, correct, resample ----------------------

def fix44(r: float) -> int:
    return int(_load().oq_fix44(float(np.float32(r))))


def scale_floor(u: float, S: int) -> int:
    return int(_load().oq_scale_floor(float(np.float32(u)), int(S)))


def accept(p, q, draft, u, mode: int = ACCEPT_SAMPLE):
    """p [B,K+1,V] f32, q [B,K,V] f32 (or None), draft [B,K] i32, u [B,K+1] f32.

    Returns (status, n_accepted [B] i32, tokens [B,K+1] i32)."""
    pa = _c(p, np.float32)
    B, K1, V = pa.shape
    K = K1 - 1
    qa = None if q is None else _c(q, np.float32)
    da = _c(draft, np.int32).reshape(B, K)
    ua = _c(u, np.float32).reshape(B, K1)
    n = np.empty((B,), np.int32)
    t = np.empty((B, K1), np.int32)
    st = _load().oq_accept(_ptr(pa), _ptr(qa), _ptr(da), _ptr(ua), B, K, V, mode,
                           _ptr(n), _ptr(t))
    if st == BAD_ARG:
        raise ValueError("oq_accept: bad arguments")
    return st, n, t


def sample(probs, u):
    """token[b] ~ probs[b,:] by the fixed-point inverse CDF; -1 if no mass."""
    pa = _c(probs, np.float32)
    B, V = pa.shape
    ua = _c(u, np.float32).reshape(B)
    t = np.empty((B,), np.int32)
    st = _load().oq_sample(_ptr(pa), _ptr(ua), B, V, _ptr(t))
    return st, t


def enum_sweep(p, q, draft, u_fixed, pos: int, grid_bits: int = 24,
               mode: int = ACCEPT_SAMPLE) -> np.ndarray:
    """Histogram of (n, token at n) over every grid value of uniform `pos`."""
    pa = _c(p, np.float32)
    K1, V = pa.shape
    K = K1 - 1
    qa = None if q is None else _c(q, np.float32)
    da = _c(draft, np.int32).reshape(K)
    ua = _c(u_fixed, np.float32).reshape(K1)
    hist = np.zeros(((K + 1) * V + 1,), np.uint64)
    st = _load().oq_enum_sweep(_ptr(pa), _ptr(qa), _ptr(da), _ptr(ua), K, V, mode, pos,
                               grid_bits, _ptr(hist))
    if st != OK:
        raise ValueError(f"oq_enum_sweep status {st}")
    return hist


# ---- probabilities from logits --------------------------------------------------

def exp_neg(x) -> np.ndarray:
    """e^x for x <= 0 by the oracle's fp32 Cody-Waite + Taylor-7 routine."""
    xs = _c(np.atleast_1d(np.asarray(x, np.float32)), np.float32)
    out = np.empty(xs.shape, np.float32)
    _load().oq_exp_neg_array(_ptr(xs), xs.size, _ptr(out))
    return out


def softmax_row(z16, T: float = 1.0) -> np.ndarray:
    """softmax(z / T) of one row of fp16 logits (bit patterns or float16)."""
    za = _c(np.asarray(z16).view(np.uint16) if np.asarray(z16).dtype == np.float16
            else z16, np.uint16)
    p = np.empty(za.shape, np.float32)
    st = _load().oq_softmax_row(_ptr(za), za.size, float(T), _ptr(p))
    if st != OK:
        raise ValueError("oq_softmax_row: bad arguments")
    return p


def accept_logits(zp, zq, draft, u, T: float = 1.0, mode: int = ACCEPT_SAMPLE):
    """zp [B,K+1,V] fp16, zq [K,B,V] fp16 (None when K == 0), draft [B,K],
    u [B,K+1] -> (status, n_accepted [B], tokens [B,K+1])."""
    za = _c(np.asarray(zp).view(np.uint16), np.uint16)
    B, K1, V = za.shape
    K = K1 - 1
    qa = None if zq is None else _c(np.asarray(zq).view(np.uint16), np.uint16)
    da = _c(draft, np.int32).reshape(B, K)
    ua = _c(u, np.float32).reshape(B, K1)
    n = np.empty((B,), np.int32)
    t = np.empty((B, K1), np.int32)
    st = _load().oq_accept_logits(_ptr(za), _ptr(qa), _ptr(da), _ptr(ua), B, K, V, float(T), mode,
                                  _ptr(n), _ptr(t))
    if st == BAD_ARG:
        raise ValueError("oq_accept_logits: bad arguments")
    return st, n, t


def sample_logits(z, u, T: float = 1.0):
    """token[b] ~ softmax(z[b,:] / T) by the fixed-point inverse CDF."""
    za = _c(np.asarray(z).view(np.uint16), np.uint16)
    B, V = za.shape
    ua = _c(u, np.float32).reshape(B)
    t = np.empty((B,), np.int32)
    st = _load().oq_sample_logits(_ptr(za), _ptr(ua), B, V, float(T), _ptr(t))
    if st == BAD_ARG:
        raise ValueError("oq_sample_logits: bad arguments")
    return st, t


# ---- the decoder around the linear stack ----------------------------------------

def rmsnorm(x, gamma, eps: float = 1e-6) -> np.ndarray:
    """y = x / sqrt(mean(x^2) + eps) * gamma in fp64; x [M, H], gamma [H]."""
    xa = _c(np.atleast_2d(x), np.float64)
    ga = _c(gamma, np.float64)
    M, H = xa.shape
    y = np.empty_like(xa)
    _load().oq_rmsnorm(_ptr(xa), _ptr(ga), M, H, float(eps), _ptr(y))
    return y


def rope(x, pos, nheads: int, head_dim: int, theta: float = 1e6) -> np.ndarray:
    """Rotary embedding (rotate-half pairs d, d + D/2) of rows x [M, nheads*D]."""
    xa = _c(np.atleast_2d(x), np.float64).copy()
    pa = _c(pos, np.int64)
    M = xa.shape[0]
    _load().oq_rope(_ptr(xa), _ptr(pa), M, nheads, head_dim, float(theta))
    return xa


def attention(q, k, v, qpos) -> np.ndarray:
    """q [T, Hq, D], k/v [L, Hkv, D]; query t sees keys 0..qpos[t] -> [T, Hq, D]."""
    qa = _c(q, np.float64)
    ka = _c(k, np.float64)
    va = _c(v, np.float64)
    T, Hq, D = qa.shape
    L, Hkv, _ = ka.shape
    pa = _c(qpos, np.int64)
    out = np.empty((T, Hq, D), np.float64)
    _load().oq_attention(_ptr(qa), _ptr(ka), _ptr(va), _ptr(pa), T, L, Hq, Hkv, D, _ptr(out))
    return out


def silu_gate_rows(gu, inter: int) -> np.ndarray:
    """silu(g) * u for rows gu = [g | u] of width 2 * inter (the fused gate/up layout)."""
    gu = np.asarray(gu, np.float64)
    return silu_gate(gu[:, :inter], gu[:, inter:])


# ---- Sec. III-D: the decoder as a function of its token sequence -----------------
#
# A plain restatement with no KV cache: every call recomputes the whole
# sequence, so the cache, its positions and its rollback on the CUDA side are
# checked against a computation that has none of them.  Model internals follow
# the Qwen2.5 decoder (the paper gives none): pre-norm layers
#   x += o(attention(rope(q), rope(k), v)),  x += down(silu(gate) * up)
# over RMSNorm'ed inputs, a final RMSNorm and the lm_head; the input
# embedding is its own fp16 table (or the lm_head's, tied, when absent).

def decoder_logits(params: dict, tokens, rows=None) -> np.ndarray:
    """Logits (fp64) of the decoder over one token sequence.

    params: 'layers' = list of (w_qkv, w_o, w_gate_up, w_down) float arrays,
    'lm_head' [V, H], 'embed' [V, H] (optional), 'gamma' = 2 L + 1 gains, 'q_heads', 'kv_heads',
    'head_dim', 'intermediate', 'eps', 'theta'.  rows: positions whose
    logits are wanted (default: all)."""
    tok = np.asarray(tokens, np.int64)
    n = len(tok)
    Hq, Hkv, D = params["q_heads"], params["kv_heads"], params["head_dim"]
    inter, eps, theta = params["intermediate"], params["eps"], params["theta"]
    emb = np.asarray(params.get("embed", params["lm_head"]), np.float64)
    lm = np.asarray(params["lm_head"], np.float64)
    gam = params["gamma"]
    pos = np.arange(n, dtype=np.int64)
    x = emb[tok].copy()
    for li, (w_qkv, w_o, w_gu, w_dn) in enumerate(params["layers"]):
        h = rmsnorm(x, gam[2 * li], eps)
        qkv = linear(h, w_qkv)
        q = rope(qkv[:, :Hq * D], pos, Hq, D, theta)
        k = rope(qkv[:, Hq * D:(Hq + Hkv) * D], pos, Hkv, D, theta)
        v = qkv[:, (Hq + Hkv) * D:]
        a = attention(q.reshape(n, Hq, D), k.reshape(n, Hkv, D), v.reshape(n, Hkv, D), pos)
        x = x + linear(a.reshape(n, Hq * D), w_o)
        h = rmsnorm(x, gam[2 * li + 1], eps)
        x = x + linear(silu_gate_rows(linear(h, w_gu), inter), w_dn)
    sel = pos if rows is None else np.asarray(rows, np.int64)
    return linear(rmsnorm(x[sel], gam[-1], eps), lm)


def generate_greedy(params: dict, prompt, n_new: int):
    """Greedy continuation of one prompt: each new token is the argmax of
    the logits at the last position given everything before it (lowest
    index on ties).  Returns (tokens, gaps), gaps[i] = the distance between
    the two largest logits at step i (how far step i is from a tie)."""
    seq = [int(t) for t in prompt]
    out, gaps = [], []
    for _ in range(n_new):
        z = decoder_logits(params, seq, rows=[len(seq) - 1])[0]
        order = np.argsort(-z, kind="stable")
        out.append(int(order[0]))
        gaps.append(float(z[order[0]] - z[order[1]]))
        seq.append(int(order[0]))
    return out, gaps


# ---- Sec. III-D.4: the bookkeeping between cycles --------------------------------

def spec_commit(n_accepted, tokens, hist, length, K: int):
    """Append tokens[b, :n+1] (n = n_accepted[b]; None = 0; n < 0 appends
    nothing) to each history, then the next cycle's positions pos [K+1, B]
    (draft step 0 at L-2, draft step k at L-1+k, verify at L-1) and the last
    two tokens.  Returns (hist, length, pos, last2, bad) as new arrays;
    `bad` marks a sequence whose history overflowed or is shorter than 2."""
    hist = [list(map(int, h)) for h in np.asarray(hist)]
    length = [int(x) for x in np.asarray(length)]
    tokens = np.asarray(tokens).reshape(len(length), -1)
    B, cap = len(length), len(hist[0])
    pos = np.zeros((K + 1, B), np.int32)
    last2 = np.zeros((B, 2), np.int32)
    bad = np.zeros(B, bool)
    for b in range(B):
        L = length[b]
        if L < 0 or L > cap:
            bad[b], L = True, 0
        else:
            n = 0 if n_accepted is None else int(n_accepted[b])
            if n >= tokens.shape[1]:
                bad[b] = True
            elif n >= 0:
                new = [int(t) for t in tokens[b, :n + 1]]
                room = cap - L
                if len(new) > room:
                    bad[b] = True
                    new = new[:room]
                hist[b][L:L + len(new)] = new
                L += len(new)
        if L < 2:
            bad[b] = True
        length[b] = L
        last2[b] = (hist[b][L - 2] if L >= 2 else -1, hist[b][L - 1] if L >= 1 else -1)
        if K >= 1:
            pos[0, b] = L - 2
        for k in range(1, K):
            pos[k, b] = L - 1 + k
        pos[K, b] = L - 1
    return np.array(hist, np.int32), np.array(length, np.int32), pos, last2, bad


def spec_drafts(samples, last2):
    """(verify tokens [B, K+1], draft [B, K]) from the draft steps' tokens
    samples [K, B] and the last committed token last2[:, 1]."""
    s = np.asarray(samples, np.int32)
    l2 = np.asarray(last2, np.int32)
    K, B = s.shape
    verify = np.concatenate([l2[:, 1:2], s.T], axis=1)
    return verify.astype(np.int32), s.T.copy()
