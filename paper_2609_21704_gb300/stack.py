"""Device-resident linear stack of a Qwen2.5-shaped model and one
speculative draft/verify cycle over it, driven through the C ABI.

Sec. III-A: one FP16 parent W16 with the INT4 (Q4) and FP8 (Q8) variants
derived from it by ``sq_quantize``, all resident in HBM at once.
Sec. III-D.2: the draft pass runs every projection plus lm_head at M = B.
Sec. III-D.3: the verify pass runs them at M = B (K + 1) with the parent.
Sec. III-D.4: ``sq_accept`` over the vocabulary.

Attention, RMSNorm, RoPE and the residual stream are outside the hot path.
A pass therefore runs, per layer:
    qkv = x_l W_qkv^T                      (fused q/k/v, one launch)
    o   = a W_o^T                          a = the first M * q_out values of
                                           qkv read as [M, q_out] (for M = 1
                                           exactly the q row): attention's
                                           stand-in keeps the qkv -> o order
    h   = silu(x_l W_g^T) * (x_l W_u^T)    (fused gate/up + SiLU, one launch)
    d   = h W_down^T
and then logits = x W_lm^T.  x_l is a resident synthetic N(0, 1) hidden
state; without normalisation a random-init residual stream overflows fp16
within a few layers, so the layers are fed fresh activations while every
projection still runs once, in stream order, with its real weights.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import (SQ_EPI_NONE, SQ_EPI_SILU_GATE, SQ_FP8_E4M3_ROW, SQ_INT4_G128, SQ_W_FP8,
               SQ_W_FP16, SQ_W_INT4, sq_linear_chain, sq_linear_ex, sq_quantize,
               sq_quantized_bytes, synth)
from .shapes import StackShape

WKIND = {"fp16": SQ_W_FP16, "int4": SQ_W_INT4, "fp8": SQ_W_FP8}
BYTES_PER_WEIGHT = {"fp16": 2.0, "int4": 0.5 + 2.0 / 128.0, "fp8": 1.0}


@dataclass
class Proj:
    name: str
    n_out: int      # weight rows
    k_in: int
    epi: int
    w16: torch.Tensor
    q: dict         # variant -> (codes, scales)

    def weight(self, variant):
        if variant == "fp16":
            return self.w16, None
        return self.q[variant]

    def y_cols(self):
        return self.n_out // 2 if self.epi == SQ_EPI_SILU_GATE else self.n_out

    def weight_bytes(self, variant) -> int:
        n, k = self.n_out, self.k_in
        if variant == "fp16":
            return 2 * n * k
        kind = SQ_INT4_G128 if variant == "int4" else SQ_FP8_E4M3_ROW
        cb, sb = sq_quantized_bytes(kind, n, k)
        return cb + sb


class LinearStack:
    """All projections of ``layers`` decoder layers plus lm_head, FP16 parent
    and the requested derived variants, resident on ``device``."""

    def __init__(self, shape: StackShape, device, seed: int = 0, variants=("int4", "fp8"),
                 layers: int | None = None, with_lm_head: bool = True, host_weights: bool = False):
        self.shape = shape
        self.device = torch.device(device)
        self.variants = tuple(variants)
        # host_weights: draw the parents with numpy on the host (small test
        # models whose weights the oracle regenerates from the same seeds)
        self.host_weights = host_weights
        self.layers = []
        nl = shape.layers if layers is None else layers
        s = seed
        for _ in range(nl):
            layer = []
            for name, n, k in shape.projections():
                epi = SQ_EPI_SILU_GATE if name == "gate_up" else SQ_EPI_NONE
                layer.append(self._make(name, n, k, epi, s))
                s += 1
            self.layers.append(layer)
        self.lm_head = None
        if with_lm_head:
            name, n, k = shape.lm_head()
            self.lm_head = self._make(name, n, k, SQ_EPI_NONE, s)
            s += 1
        self._embed_seed = s
        self._embed = None

    def embedding(self) -> torch.Tensor:
        """The input embedding, fp16 [vocab, hidden]: its own seeded table
        (untied from the lm_head), drawn on first use and shared by the
        parent and its variants (only the linear layers are quantised)."""
        if self._embed is None:
            sh = self.shape
            ws = synth.stack_weight_seed(self._embed_seed, 0)
            if self.host_weights:
                self._embed = torch.from_numpy(synth.weights_fp16(ws, sh.vocab, sh.hidden)).to(self.device)
            else:
                self._embed = synth.weights_fp16_device(ws, sh.vocab, sh.hidden, self.device)
        return self._embed

    def _make(self, name, n, k, epi, seed) -> Proj:
        ws = synth.stack_weight_seed(seed, 0)
        if self.host_weights:
            w16 = torch.from_numpy(synth.weights_fp16(ws, n, k)).to(self.device)
        else:
            w16 = synth.weights_fp16_device(ws, n, k, self.device)
        q = {}
        for v in self.variants:
            kind = SQ_INT4_G128 if v == "int4" else SQ_FP8_E4M3_ROW
            cb, sb = sq_quantized_bytes(kind, n, k)
            codes = torch.empty((n, cb // n), dtype=torch.uint8, device=self.device)
            if v == "int4":
                scales = torch.empty((n, k // 128), dtype=torch.float16, device=self.device)
            else:
                scales = torch.empty((n,), dtype=torch.float32, device=self.device)
            sq_quantize(w16, kind, codes, scales)
            q[v] = (codes, scales)
        return Proj(name, n, k, epi, w16, q)

    def projections(self):
        for layer in self.layers:
            yield from layer
        if self.lm_head is not None:
            yield self.lm_head

    def launches_per_pass(self) -> int:
        return sum(1 for _ in self.projections())

    def weight_bytes(self, variant) -> int:
        return sum(p.weight_bytes(variant) for p in self.projections())

    def activation_bytes(self, M: int) -> int:
        return sum(2 * M * (p.k_in + p.y_cols()) for p in self.projections())

    def params(self) -> int:
        return sum(p.n_out * p.k_in for p in self.projections())


class PassBuffers:
    """Activations and outputs of one pass at M rows."""

    def __init__(self, stack: LinearStack, M: int, seed: int = 1):
        sh, dev = stack.shape, stack.device
        self.M = M
        self.x = synth.activations_fp16_device(seed, M, sh.hidden, dev)
        nq = sh.q_out + 2 * sh.kv_out
        self.qkv = torch.empty((M, nq), dtype=torch.float16, device=dev)
        self.o = torch.empty((M, sh.hidden), dtype=torch.float16, device=dev)
        self.h = torch.empty((M, sh.intermediate), dtype=torch.float16, device=dev)
        self.d = torch.empty((M, sh.hidden), dtype=torch.float16, device=dev)
        self.logits = torch.empty((M, sh.vocab), dtype=torch.float16, device=dev) \
            if stack.lm_head is not None else None
        # attention stand-in: the first M * q_out values of qkv as [M, q_out]
        self.attn = self.qkv.view(-1)[: M * sh.q_out].view(M, sh.q_out)


def pass_ops(stack: LinearStack, variant: str, b: PassBuffers, logits=None):
    """The linear calls of one pass in decoder order, as sq_linear_chain ops;
    `logits` (fp16 [M, vocab]) replaces b.logits as the lm_head output."""
    wk = WKIND[variant]
    ops = []
    for layer in stack.layers:
        qkv, o, gu, down = layer
        ops.append((wk, b.x, *qkv.weight(variant), None, None, SQ_EPI_NONE, b.qkv))
        ops.append((wk, b.attn, *o.weight(variant), None, None, SQ_EPI_NONE, b.o))
        ops.append((wk, b.x, *gu.weight(variant), None, None, SQ_EPI_SILU_GATE, b.h))
        ops.append((wk, b.h, *down.weight(variant), None, None, SQ_EPI_NONE, b.d))
    if stack.lm_head is not None:
        ops.append((wk, b.x, *stack.lm_head.weight(variant), None, None, SQ_EPI_NONE,
                    b.logits if logits is None else logits))
    return ops


def run_pass(stack: LinearStack, variant: str, b: PassBuffers, stream=None, logits=None) -> None:
    """One draft (variant int4/fp8) or verify (fp16, or fp8) pass: every
    projection of every layer plus lm_head, in decoder order, as one
    sq_linear_chain call."""
    sq_linear_chain(pass_ops(stack, variant, b, logits), stream)


def run_pass_unchained(stack: LinearStack, variant: str, b: PassBuffers, stream=None,
                       logits=None) -> None:
    """The same pass as separate sq_linear_ex calls."""
    for (wk, x, w, s, bias, res, epi, y) in pass_ops(stack, variant, b, logits):
        sq_linear_ex(wk, x, w, s, bias, res, epi, y, stream)


# ---- the decoder step around the linear stack ---------------------------------------

HEAD_DIM = 128
ROPE_THETA = 1e6       # Qwen2.5
RMS_EPS = 1e-6


class DecoderState:
    """Per-model state of a decoder pass over T new tokens of B sequences: a
    KV cache per layer ([B, Hkv, max_ctx, 128] fp16, keys rotated), the
    RMSNorm gains, the residual stream and the pass's activations.  Token t
    of sequence b sits at position pos0[b] + t.  `share` gives another
    state whose caches and gains this one uses (states of one model at
    different T); `share_gains` gives only the gains (a second model)."""

    def __init__(self, stack: LinearStack, B: int, T: int, max_ctx: int, context: int = 0,
                 seed: int = 5, share: "DecoderState | None" = None,
                 share_gains: "DecoderState | None" = None):
        from . import sq_attention_workspace_bytes
        sh, dev = stack.shape, stack.device
        self.B, self.T, self.max_ctx = B, T, max_ctx
        nl = len(stack.layers)
        if share is not None:
            assert share.B == B and share.max_ctx == max_ctx
            self.k, self.v = share.k, share.v
        else:
            cache = (B, sh.kv_heads, max_ctx, HEAD_DIM)
            self.k = [torch.zeros(cache, dtype=torch.float16, device=dev) for _ in range(nl)]
            self.v = [torch.zeros(cache, dtype=torch.float16, device=dev) for _ in range(nl)]
        src = share if share is not None else share_gains
        if src is not None:
            self.gamma = src.gamma
        else:
            self.gamma = [torch.from_numpy(g).to(dev) for g in synth.rms_gains(seed, sh.hidden, 2 * nl + 1)]
        self.pos0 = torch.full((B,), context, dtype=torch.int32, device=dev)
        M = B * T
        self.x = synth.activations_fp16_device(seed + 99, M, sh.hidden, dev)
        self.h = torch.empty((M, sh.hidden), dtype=torch.float16, device=dev)
        self.qkv = torch.empty((M, sh.q_out + 2 * sh.kv_out), dtype=torch.float16, device=dev)
        self.attn = torch.empty((M, sh.q_out), dtype=torch.float16, device=dev)
        self.g = torch.empty((M, sh.intermediate), dtype=torch.float16, device=dev)
        self.logits = torch.empty((M, sh.vocab), dtype=torch.float16, device=dev) \
            if stack.lm_head is not None else None
        # the last token of each sequence, for passes whose lm_head reads only it
        self.last_rows = torch.arange(B, dtype=torch.int32, device=dev) * T + (T - 1)
        self.x_last = torch.empty((B, sh.hidden), dtype=torch.float16, device=dev)
        self.ws = torch.empty(sq_attention_workspace_bytes(B, T, sh.q_heads, sh.kv_heads, max_ctx),
                              dtype=torch.uint8, device=dev)


def decoder_pass(stack: LinearStack, variant: str, st: DecoderState, stream=None,
                 logits=None, pos0=None, last_only: bool = False, with_logits: bool = True,
                 fused: bool = True, fuse_norm: bool | None = None, fuse_append: bool | None = None) -> None:
    """One decoder step (draft or verify) with the variant's weights: per
    layer x += o(attn(rope(qkv(norm(x))))), x += down(silu-gate(norm(x)));
    then logits = lm_head(norm(x)) (into `logits` when given).  The new
    tokens' keys and values are appended to the caches before attention
    reads them.  pos0 (int32 [B], device) overrides st.pos0; last_only
    runs the lm_head on each sequence's last token only (logits [B, V]);
    with_logits=False stops after the layers (a prefill that only fills
    the cache).  fused: each RMSNorm runs inside the projection that reads
    it (sq_linear_norm) and, for one new token per sequence, the cache
    append inside the attention (sq_attention_append): six launches per
    layer instead of nine; the results are bit-identical either way
    (fuse_norm / fuse_append override the two choices)."""
    from . import (SQ_EPI_RESIDUAL, sq_attention, sq_attention_append, sq_embed, sq_kv_append,
                   sq_linear_norm, sq_rmsnorm)
    sh = stack.shape
    wk = WKIND[variant]
    B, T = st.B, st.T
    pos = st.pos0 if pos0 is None else pos0
    fuse_norm = fused if fuse_norm is None else fuse_norm
    # the fused append measured faster in passes of one new token per
    # sequence but slower from two on (the kernels launched after it lose
    # overlap; 10 us per layer at five tokens), so it is the default at T = 1
    fuse_append = (fused and T == 1) if fuse_append is None else fuse_append

    def normed(x, gamma, h, w, s, epi, y):
        if fuse_norm:
            sq_linear_norm(wk, x, gamma, RMS_EPS, h, w, s, None, None, epi, y, stream)
        else:
            sq_rmsnorm(x, gamma, RMS_EPS, h, stream)
            sq_linear_ex(wk, h, w, s, None, None, epi, y, stream)

    for li, (qkv, o, gu, down) in enumerate(stack.layers):
        w, s = qkv.weight(variant)
        normed(st.x, st.gamma[2 * li], st.h, w, s, SQ_EPI_NONE, st.qkv)
        if fuse_append:
            sq_attention_append(st.qkv, B, T, sh.q_heads, sh.kv_heads, pos, ROPE_THETA, st.k[li], st.v[li],
                                st.attn, st.ws, stream)
        else:
            sq_kv_append(st.qkv, B, T, sh.q_heads, sh.kv_heads, pos, ROPE_THETA, st.k[li], st.v[li], stream)
            sq_attention(st.qkv, B, T, sh.q_heads, sh.kv_heads, pos, ROPE_THETA, st.k[li], st.v[li],
                         st.attn, st.ws, stream)
        w, s = o.weight(variant)
        sq_linear_ex(wk, st.attn, w, s, None, st.x, SQ_EPI_RESIDUAL, st.x, stream)
        w, s = gu.weight(variant)
        normed(st.x, st.gamma[2 * li + 1], st.h, w, s, SQ_EPI_SILU_GATE, st.g)
        w, s = down.weight(variant)
        sq_linear_ex(wk, st.g, w, s, None, st.x, SQ_EPI_RESIDUAL, st.x, stream)
    if stack.lm_head is None or not with_logits:
        return
    x, h = st.x, st.h
    if last_only and T > 1:
        sq_embed(st.last_rows, st.x, st.x_last, stream)   # row gather
        x, h = st.x_last, st.h[:B]
    w, s = stack.lm_head.weight(variant)
    normed(x, st.gamma[-1], h, w, s, SQ_EPI_NONE, st.logits if logits is None else logits)
