"""Speculative generation on the device (Sec. III-D), and direct decoding
with the parent for comparison (K = 0).

The derived variant (INT4 or FP8) and the FP16 parent are the two models of
one stack; each keeps its own KV cache, and both share the RMSNorm gains and
the fp16 input embedding (only the linear layers are quantised).  One cycle:

  draft step 0      feed the last two committed tokens (T = 2, positions
                    L-2, L-1); the second-last is fed again because its key
                    and value are missing from the draft cache when every
                    draft of the previous cycle was accepted
  draft steps 1..K-1  feed the previous draft token (T = 1)
                    after each step, one token from the draft logits
                    (argmax, or a draw with the caller's uniform)
  verify            the parent over (last token, d_1 .. d_K), T = K + 1
  accept            Sec. III-D.4 on both sets of logits
  commit            append the n + 1 new tokens, derive next positions

Every step, the bookkeeping included, runs in the library's kernels, so a
cycle is one CUDA graph replay with no host synchronisation; sequences
advance by their own n_b + 1 tokens with per-sequence positions, and stale
cache entries past a sequence's length are never read (attention stops at
each query's own position) and are overwritten by the next cycle.
"""
from __future__ import annotations

import numpy as np
import torch

from . import (SQ_ACCEPT_GREEDY, SQ_ACCEPT_SAMPLE, sq_accept_logits, sq_accept_logits_workspace_bytes,
               sq_check, sq_embed, sq_sample_logits, sq_spec_commit, sq_spec_drafts, synth)
from .stack import DecoderState, LinearStack, decoder_pass

# Limits of one sq_attention call (see its declaration): at most 32 new
# tokens per sequence, and (Hq / Hkv) * T <= 200 queries per key/value head.
ATTN_MAX_T = 32
ATTN_MAX_GROUP_QUERIES = 200


# Rows of one linear call (sq_linear_ex): B sequences x T tokens of a pass.
LINEAR_MAX_ROWS = 256


def prefill_chunk(q_heads: int, kv_heads: int, B: int = 1) -> int:
    """Tokens per prefill pass: as many as one attention call takes, and at
    most LINEAR_MAX_ROWS rows over the B sequences."""
    return max(1, min(ATTN_MAX_T, ATTN_MAX_GROUP_QUERIES // (q_heads // kv_heads), LINEAR_MAX_ROWS // B))


class Generator:
    """Generation for B sequences over `stack` (which must hold the draft
    variant and an lm_head).  K >= 1: speculative cycles with `draft`
    drafting and `verifier` verifying; K = 0: direct decoding with
    `verifier`, one token per cycle."""

    def __init__(self, stack: LinearStack, B: int, K: int, prompt_len: int, max_ctx: int,
                 draft: str = "int4", verifier: str = "fp16", mode: int = SQ_ACCEPT_GREEDY,
                 temperature: float = 1.0, seed: int = 0):
        if stack.lm_head is None:
            raise ValueError("generation needs the lm_head")
        if K < 0 or K > 16 or prompt_len < 1:
            raise ValueError("need 0 <= K <= 16 and a prompt of at least one token")
        if prompt_len + 1 + K > max_ctx:
            raise ValueError("max_ctx too small for the prompt and one cycle")
        sh, dev = stack.shape, stack.device
        self.stack, self.B, self.K, self.P, self.max_ctx = stack, B, K, prompt_len, max_ctx
        self.draft, self.verifier, self.mode, self.temperature = draft, verifier, mode, temperature
        self.seed = seed
        V = sh.vocab
        self.table = stack.embedding()            # input embedding [V, H]
        i32 = dict(dtype=torch.int32, device=dev)

        # one cache per model; states per T share it
        self.tv = DecoderState(stack, B, K + 1, max_ctx, seed=seed + 5)
        self.d2 = self.d1 = None
        if K > 0:
            self.d2 = DecoderState(stack, B, 2, max_ctx, share_gains=self.tv)
            if K > 1:
                self.d1 = DecoderState(stack, B, 1, max_ctx, share=self.d2)
        pc = prefill_chunk(sh.q_heads, sh.kv_heads, B)
        self.chunks = [(s, min(pc, prompt_len - s)) for s in range(0, prompt_len, pc)]
        self.pre_t, self.pre_d = {}, {}
        for _, T in self.chunks:
            if T not in self.pre_t:
                self.pre_t[T] = DecoderState(stack, B, T, max_ctx, share=self.tv)
                if K > 0:
                    self.pre_d[T] = DecoderState(stack, B, T, max_ctx, share=self.d2)
        self.chunk_pos = {s: torch.full((B,), s, **i32) for s, _ in self.chunks}

        # token state on the device
        self.hist = torch.zeros((B, max_ctx), **i32)
        self.len = torch.zeros((B,), **i32)
        self.pos = torch.zeros((K + 1, B), **i32)
        self.last2 = torch.zeros((B, 2), **i32)
        kk = max(K, 1)
        self.samples = torch.zeros((kk, B), **i32)
        self.verify_in = torch.zeros((B, K + 1), **i32)
        self.draft_tok = torch.zeros((B, kk), **i32)
        self.n = torch.zeros((B,), **i32)
        self.n_pick = torch.zeros((B,), **i32)      # the greedy pick's (unused) accepted count
        self.tok = torch.zeros((B, K + 1), **i32)
        self.tok1 = torch.zeros((B, 1), **i32)
        self.zq = torch.empty((kk, B, V), dtype=torch.float16, device=dev)
        self.z1 = torch.empty((B, V), dtype=torch.float16, device=dev)
        self.zp = self.tv.logits.view(B, K + 1, V)
        self.u_draft = torch.zeros((kk, B), dtype=torch.float32, device=dev)
        self.u_acc = torch.zeros((B, K + 1), dtype=torch.float32, device=dev)
        self.u1 = torch.zeros((B, 1), dtype=torch.float32, device=dev)
        self.ws_pick = torch.zeros(sq_accept_logits_workspace_bytes(B, 0, V), dtype=torch.uint8, device=dev)
        self.ws_acc = torch.zeros(sq_accept_logits_workspace_bytes(B, K, V), dtype=torch.uint8, device=dev)
        self._graph = None
        self._cycles = 0

    # ---- steps ------------------------------------------------------------------
    def _pick(self, z, u, out, stream):
        """One token per sequence from fp16 logits z [B, V] into out (int32, B)."""
        if self.mode == SQ_ACCEPT_GREEDY:
            sq_accept_logits(z.view(self.B, 1, -1), None, None, u, self.temperature, SQ_ACCEPT_GREEDY,
                             self.n_pick, out, self.ws_pick, stream)
        else:
            sq_sample_logits(z, u, self.temperature, out, self.ws_pick, stream)

    def max_cycles(self) -> int:
        """Cycles that always fit the cache: each adds at most K + 1 tokens
        and the verify pass writes K positions past the committed length."""
        return (self.max_ctx - self.K - self.P - 1) // (self.K + 1)

    def prefill(self, prompt: np.ndarray, stream: torch.cuda.Stream) -> None:
        """Both models read the prompt (int32 [B, P]) into their caches; the
        parent's last-token logits give the first generated token."""
        B, P = self.B, self.P
        prompt = np.ascontiguousarray(prompt, dtype=np.int32)
        if prompt.shape != (B, P):
            raise ValueError(f"prompt shape {prompt.shape} != {(B, P)}")
        dev = self.stack.device
        self._cycles = 0
        with torch.cuda.stream(stream):
            ids = torch.from_numpy(prompt).to(dev)
            self.hist.zero_()
            self.hist[:, :P] = ids
            self.len.fill_(P)
            for s, T in self.chunks:
                chunk = ids[:, s:s + T].contiguous()
                last = s + T == P
                st = self.pre_t[T]
                sq_embed(chunk, self.table, st.x, stream)
                decoder_pass(self.stack, self.verifier, st, stream, logits=self.z1, pos0=self.chunk_pos[s],
                             last_only=True, with_logits=last)
                if self.K > 0:
                    sd = self.pre_d[T]
                    sq_embed(chunk, self.table, sd.x, stream)
                    decoder_pass(self.stack, self.draft, sd, stream, pos0=self.chunk_pos[s],
                                 with_logits=False)
            self.u1.copy_(torch.from_numpy(synth.uniforms(self.seed ^ 0x9F1, (B, 1))).to(dev))
            self._pick(self.z1, self.u1, self.tok1, stream)
            sq_spec_commit(None, self.tok1, self.hist, self.len, self.pos, self.last2, self.K, stream)

    def cycle(self, stream=None) -> None:
        """One draft / verify / accept / commit cycle (K >= 1), or one direct
        decoding step (K = 0)."""
        K, B, stk = self.K, self.B, self.stack
        if K == 0:
            tv = self.tv
            # the last committed token of each sequence: last2[b, 1]
            sq_embed(self.last2.view(-1)[1:], self.table, tv.x, stream, ids_stride=2, M=B)
            decoder_pass(stk, self.verifier, tv, stream, pos0=self.pos[0])
            self._pick(tv.logits, self.u_acc, self.tok1, stream)
            sq_spec_commit(None, self.tok1, self.hist, self.len, self.pos, self.last2, 0, stream)
            return
        d2 = self.d2
        sq_embed(self.last2, self.table, d2.x, stream)
        decoder_pass(stk, self.draft, d2, stream, logits=self.zq[0], pos0=self.pos[0], last_only=True)
        self._pick(self.zq[0], self.u_draft[0], self.samples[0], stream)
        for k in range(1, K):
            d1 = self.d1
            sq_embed(self.samples[k - 1], self.table, d1.x, stream)
            decoder_pass(stk, self.draft, d1, stream, logits=self.zq[k], pos0=self.pos[k])
            self._pick(self.zq[k], self.u_draft[k], self.samples[k], stream)
        sq_spec_drafts(self.samples, self.last2, self.verify_in, self.draft_tok, stream)
        sq_embed(self.verify_in, self.table, self.tv.x, stream)
        decoder_pass(stk, self.verifier, self.tv, stream, pos0=self.pos[K])
        sq_accept_logits(self.zp, self.zq, self.draft_tok, self.u_acc, self.temperature, self.mode,
                         self.n, self.tok, self.ws_acc, stream)
        sq_spec_commit(self.n, self.tok, self.hist, self.len, self.pos, self.last2, K, stream)

    # ---- driving ----------------------------------------------------------------
    def _draws(self, c0: int, cycles: int):
        """The uniforms of cycles c0 .. c0+cycles-1 (sampling mode), seeded
        per cycle and moved to the device in one copy; each cycle's slice is
        copied into the buffers the captured cycle reads."""
        kk = self.u_draft.shape[0]
        ud = np.stack([synth.uniforms(self.seed * 1000003 + 2 * c + 1, (kk, self.B))
                       for c in range(c0, c0 + cycles)])
        ua = np.stack([synth.uniforms(self.seed * 1000003 + 2 * c + 2, (self.B, self.K + 1))
                       for c in range(c0, c0 + cycles)])
        dev = self.stack.device
        return torch.from_numpy(ud).to(dev), torch.from_numpy(ua).to(dev)

    def run(self, cycles: int, stream: torch.cuda.Stream, graph: bool = True) -> None:
        """`cycles` more cycles on `stream`.  With graph=True the first cycle
        this generator runs is eager (and then captured); every later one is
        a replay of that CUDA graph (the buffers it reads never move)."""
        if self._cycles + cycles > self.max_cycles():
            raise ValueError(f"{self._cycles + cycles} cycles exceed the cache ({self.max_cycles()})")
        with torch.cuda.stream(stream):
            draws = self._draws(self._cycles, cycles) if self.mode == SQ_ACCEPT_SAMPLE else None
            for i in range(cycles):
                if draws is not None:
                    self.u_draft.copy_(draws[0][i])
                    self.u_acc.copy_(draws[1][i])
                if graph and self._graph is not None:
                    self._graph.replay()
                else:
                    self.cycle(stream)
                    if graph:
                        stream.synchronize()
                        g = torch.cuda.CUDAGraph()
                        with torch.cuda.graph(g, stream=stream):
                            self.cycle(stream)
                        self._graph = g
                self._cycles += 1

    def tokens(self) -> list:
        """The committed tokens of each sequence (prompt included)."""
        torch.cuda.synchronize()
        h = self.hist.cpu().numpy()
        n = self.len.cpu().numpy()
        return [h[b, :n[b]].tolist() for b in range(self.B)]

    def status(self) -> int:
        return sq_check()
