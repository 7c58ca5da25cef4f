"""A whole edit session on the device: verification steps and the Reuse <->
Generate controller in one captured loop.

EfficientEdit (arXiv 2506.02780) Sec. III-A alternates Reuse (the remaining
original code is the draft) and Generate (a draft model proposes edited
content, after which prefix matching finds where reuse resumes).  Here every
step's tree holds both: one reuse chain per match point of the committed
suffix in the code not yet verified, plus a generated branch.  ``EditSession``
owns the controller state -- committed tokens, tail, cursor, root token,
context length -- on the device and issues, per step, on one stream:

    ee_match_reuse -> ee_build_reuse_tree -> ee_tree_prepare
        -> target forward (caller's: q, tree K/V, hidden states)
        -> L x ee_tree_verify_attn -> ee_lmhead_accept -> ee_kv_compact
        -> context length copy -> ee_advance

``capture(k)`` records k such steps into one CUDA graph, so a replay runs k
steps with no host involvement.  The target model's layers (which produce q,
the tree's K/V and the hidden states from the draft tokens) and the draft
model are not part of this library: ``target_forward(session)`` and
``draft_proposal(session)`` are callables that write the step's inputs into the
session's buffers with device work only (capturable).
"""
from __future__ import annotations

import math

import torch

from . import (EE_HEAD_DIM, ee_advance, ee_build_reuse_tree, ee_kv_compact, ee_lmhead_accept, ee_match_reuse,
               ee_tree_prepare, ee_tree_verify_attn, new_workspace)


class EditSession:
    """Device-resident state of B edit sessions of one target model.

    orig_tokens int32 [sum len_c] / orig_off int64 [B+1]: the codes to edit.
    committed: list of B int lists, the tokens committed so far (at least n).
    k_cache / v_cache [L, num_pages, n_kv, 16, 128] bf16 holding the committed
    tokens' K/V (positions 0 .. ctx0 - 1); block_table int32 [B, max_pages]
    with pages for every position the session may reach; lm_w [V, H] bf16.
    Tree shape per step: 1 + n_branches * chain_len + gen_len nodes.
    """

    def __init__(self, *, orig_tokens, orig_off, committed, ctx_len, k_cache, v_cache, block_table, lm_w, n_q,
                 n=4, chain_len=24, n_branches=2, gen_len=4, max_matches=8, cap=None, target_forward=None,
                 draft_proposal=None, max_ctx=None):
        dev = k_cache.device
        i32 = dict(dtype=torch.int32, device=dev)
        self.B = orig_off.numel() - 1
        self.L, _, self.n_kv, page, d = k_cache.shape
        if d != EE_HEAD_DIM or page != 16:
            raise ValueError("cache layout [L, pages, n_kv, 16, 128] expected")
        self.n_q, self.n = n_q, n
        self.chain_len, self.n_branches, self.gen_len = chain_len, n_branches, gen_len
        self.T = 1 + n_branches * chain_len + gen_len
        self.total = self.B * self.T
        self.max_matches = max_matches
        self.orig_tokens, self.orig_off = orig_tokens, orig_off
        self.k_cache, self.v_cache, self.block_table, self.lm_w = k_cache, v_cache, block_table, lm_w
        self.hidden_dim = lm_w.shape[1]
        self.scale = 1.0 / math.sqrt(d)
        self.max_ctx = int(max_ctx if max_ctx is not None else block_table.shape[1] * 16 - self.T)
        cap = cap or max(len(c) for c in committed) + 4096
        self.out_tok = torch.zeros((self.B, cap), **i32)
        self.out_len = torch.zeros(self.B, **i32)
        self.tail = torch.zeros((self.B, n), **i32)
        self.cursor = torch.zeros(self.B, **i32)
        self.last_tok = torch.zeros(self.B, **i32)
        for s, c in enumerate(committed):
            if len(c) < n:
                raise ValueError("each session needs at least n committed tokens")
            self.out_tok[s, :len(c)] = torch.as_tensor(c, dtype=torch.int32)
            self.out_len[s] = len(c)
            self.tail[s] = torch.as_tensor(c[-n:], dtype=torch.int32)
            self.last_tok[s] = int(c[-1])
        self.ctx_len = torch.as_tensor(ctx_len, **i32).clone()
        self.ctx_out = torch.zeros(self.B, **i32)
        # per-step buffers
        self.match_pos = torch.empty((self.B, max_matches), **i32)
        self.n_matches = torch.empty(self.B, **i32)
        self.draft_tok = torch.empty(self.total, **i32)
        self.parent = torch.empty(self.total, **i32)
        self.node_off = torch.empty(self.B + 1, **i32)
        self.cpos = torch.empty(self.total, **i32)
        self.gen_mask = torch.empty(self.total, dtype=torch.uint8, device=dev)
        self.gen_tok = torch.zeros((self.B, max(gen_len, 1)), **i32)
        self.depth = torch.empty(self.total, **i32)
        self.anc = torch.empty((self.total, 2), dtype=torch.int64, device=dev)
        bf = dict(dtype=torch.bfloat16, device=dev)
        self.q = torch.zeros((self.L, self.total, n_q, d), **bf)
        self.k_tree = torch.zeros((self.L, self.total, self.n_kv, d), **bf)
        self.v_tree = torch.zeros((self.L, self.total, self.n_kv, d), **bf)
        self.hidden = torch.zeros((self.total, self.hidden_dim), **bf)
        self.attn_out = torch.empty((self.total, n_q, d), dtype=torch.float32, device=dev)
        self.argmax = torch.empty(self.total, **i32)
        self.accept_len = torch.empty(self.B, **i32)
        self.path = torch.empty((self.B, self.T), **i32)
        self.bonus = torch.empty(self.B, **i32)
        self.dst_slot = torch.empty((self.B, self.T), **i32)
        self.ws = new_workspace(self.B, self.total, n_q, self.max_ctx, device=dev)
        self.target_forward = target_forward
        self.draft_proposal = draft_proposal
        self.graph = None
        self.graph_steps = 0

    def step(self, stream=None):
        """Enqueue one whole step: draft tree, verification, commit."""
        ee_match_reuse(self.orig_tokens, self.orig_off, self.tail, self.cursor, self.max_matches, self.match_pos,
                       self.n_matches, self.ws, stream)
        if self.gen_len and self.draft_proposal is not None:
            self.draft_proposal(self)
        ee_build_reuse_tree(self.orig_tokens, self.orig_off, self.match_pos, self.n_matches, self.last_tok, self.n,
                            self.chain_len, self.n_branches, self.draft_tok, self.parent, self.node_off, self.cpos,
                            self.gen_mask, self.ws, gen_tok=self.gen_tok if self.gen_len else None,
                            stream=stream)
        ee_tree_prepare(self.parent, self.node_off, self.depth, self.anc, self.ws, stream)
        if self.target_forward is not None:
            self.target_forward(self)
        for l in range(self.L):
            ee_tree_verify_attn(self.q[l], self.k_tree[l], self.v_tree[l], self.k_cache[l], self.v_cache[l],
                                self.block_table, self.ctx_len, self.max_ctx, self.node_off, self.anc, self.T,
                                self.scale, self.attn_out, self.ws, stream)
        ee_lmhead_accept(self.hidden, self.lm_w, self.draft_tok, self.parent, self.depth, self.anc, self.node_off,
                         self.T, self.argmax, self.accept_len, self.path, self.bonus, self.ws, stream=stream)
        ee_kv_compact(self.k_tree, self.v_tree, self.k_cache, self.v_cache, self.block_table, self.ctx_len,
                      self.ctx_out, self.node_off, self.path, self.accept_len, self.dst_slot, self.ws, stream)
        self.ctx_len.copy_(self.ctx_out)
        ee_advance(self.out_tok, self.out_len, self.draft_tok, self.cpos, self.node_off, self.path, self.accept_len,
                   self.bonus, self.tail, self.cursor, self.last_tok, self.ws, stream)

    def capture(self, steps, stream):
        """Record `steps` whole steps into one CUDA graph on `stream` (a side stream).
        Capturing runs nothing; replay() runs them."""
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            with torch.cuda.graph(g, stream=stream):
                for _ in range(steps):
                    self.step(stream)
        self.graph, self.graph_steps = g, steps
        return g

    def replay(self):
        self.graph.replay()

    def launches_per_step(self) -> int:
        """libee kernels per step: match, tree build, prepare, L attention, LM head,
        compaction, commit."""
        return 3 + self.L + 3
