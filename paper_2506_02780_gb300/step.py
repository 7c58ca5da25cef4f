"""One whole verification step as a fixed sequence of libee calls.

EfficientEdit (arXiv 2506.02780) Sec. III-A: the target scores a draft (here a
tree: reuse chain + generated branches) in one pass and keeps the longest
prefix its greedy choice agrees with.  ``VerifyStep`` owns the device output
buffers and the workspace and issues, on one stream:

    ee_match_reuse -> ee_tree_prepare -> L x ee_tree_verify_attn
        -> ee_lmhead_accept -> ee_kv_compact

or, with ``inplace_kv``, ee_tree_verify_attn_inplace and ee_kv_compact_inplace
over tree K/V that sit in the cache after each sequence's context; with
``chain`` (linear drafts of up to 2048 tokens, long reuse drafts), no tree
preparation, ee_chain_verify_attn, ee_lmhead_accept without ancestor masks and
ee_kv_compact_inplace.

No arithmetic happens here; every step runs in libee's kernels.  The whole
sequence can be captured into a CUDA graph (``capture``).
"""
from __future__ import annotations

import math

import torch

from . import (EE_HEAD_DIM, ee_chain_verify_attn, ee_kv_compact, ee_kv_compact_inplace, ee_lmhead_accept,
               ee_lmhead_accept_packed, ee_lmhead_pack_weights, ee_lmhead_packed_bytes, ee_lmhead_verify,
               ee_match_reuse, ee_tree_prepare, ee_tree_verify_attn, ee_tree_verify_attn_inplace, new_workspace)


class VerifyStep:
    """Device-resident state for repeated verification steps of one batch.

    All tensors are CUDA tensors: int32 unless noted; ``orig_off`` int64;
    q [L, total, n_q, 128], k_tree/v_tree [L, total, n_kv, 128],
    k_cache/v_cache [L, num_pages, n_kv, 16, 128], hidden [total, H],
    lm_w [V, H] in bf16.  ``max_ctx`` bounds ctx_len (host-side value).
    ``verify`` = (mode, k) switches the LM head to ee_lmhead_verify with that
    rule for the edit content marked by ``gen_mask`` (uint8 [total]); None
    keeps the greedy ee_lmhead_accept.  ``inplace_kv`` verifies with the tree's
    K/V in the cache at positions ctx + i (in-place speculative K/V): at set-up
    they are copied there from k_tree / v_tree, where a K/V projection would
    have written them, and the block table gets the columns max_ctx + max_T
    positions need (-1 padded).  ``packed_lm`` (default) rearranges lm_w once,
    at set-up, into the LM head's tile order (ee_lmhead_pack_weights, a model-
    load step, not part of a verification step) and runs the greedy LM head on
    that copy (ee_lmhead_accept_packed: bit-identical results); ``lm_packed``
    passes an already packed copy instead.
    """

    def __init__(self, *, orig_tokens, orig_off, tail, cursor, parent, node_off, draft_tok, ctx_len,
                 block_table, q, k_tree, v_tree, k_cache, v_cache, hidden, lm_w, max_ctx, max_T,
                 max_matches=8, scale=None, keep_layers=True, verify=None, gen_mask=None, inplace_kv=False,
                 chain=False, packed_lm=True, lm_packed=None):
        self.inp = dict(orig_tokens=orig_tokens, orig_off=orig_off, tail=tail, cursor=cursor,
                        parent=parent, node_off=node_off, draft_tok=draft_tok, ctx_len=ctx_len,
                        block_table=block_table, q=q, k_tree=k_tree, v_tree=v_tree, k_cache=k_cache,
                        v_cache=v_cache, hidden=hidden, lm_w=lm_w)
        dev = q.device
        self.L, self.total, self.n_q, d = q.shape
        if d != EE_HEAD_DIM:
            raise ValueError("head_dim must be 128")
        self.B = node_off.numel() - 1
        self.max_T = int(max_T)
        self.max_ctx = int(max_ctx)
        self.max_matches = int(max_matches)
        self.scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
        i32 = dict(dtype=torch.int32, device=dev)
        # the step's results are views of one int32 buffer (``outputs``; each view
        # starts on a 64-byte boundary, ``out_layout`` = name -> (offset, shape)),
        # so one device-to-host copy returns all of them
        specs = (("match_pos", (self.B, self.max_matches)), ("n_matches", (self.B,)), ("argmax", (self.total,)),
                 ("accept_len", (self.B,)), ("path", (self.B, self.max_T)), ("bonus", (self.B,)),
                 ("ctx_out", (self.B,)))
        sizes = [math.prod(sh) for _, sh in specs]
        self.outputs = torch.empty(sum(-(-n // 16) * 16 for n in sizes), **i32)
        self.out_layout = {}
        off = 0
        for (name, sh), n in zip(specs, sizes):
            setattr(self, name, self.outputs[off:off + n].view(sh))
            self.out_layout[name] = (off, sh)
            off += -(-n // 16) * 16
        self.depth = torch.empty(self.total, **i32)
        self.anc = torch.empty((self.total, 2), dtype=torch.int64, device=dev)
        n_out = self.L if keep_layers else 1
        self.attn_out = torch.empty((n_out, self.total, self.n_q, d), dtype=torch.float32, device=dev)
        self.dst_slot = torch.empty((self.B, self.max_T), **i32)
        self.ws = new_workspace(self.B, self.total, self.n_q, self.max_ctx, device=dev)
        self.verify = None if verify is None else (verify[0], int(verify[1]))
        self.gen_mask = gen_mask
        if self.verify is not None:
            k = self.verify[1]
            self.topk_ids = torch.empty((self.total, k), **i32)
            self.top_tau = torch.empty(self.total, **i32)
            self.h_norm = torch.empty(self.total, dtype=torch.float32, device=dev)
        self.chain = bool(chain)
        if self.chain and self.verify is not None:
            raise ValueError("the verification rules take trees; linear drafts are greedy")
        self.inplace_kv = bool(inplace_kv) or self.chain
        if self.inplace_kv:
            self._place_tree_kv()
        self.lm_packed = lm_packed   # tile-ordered weights to share with another step, or None
        if self.lm_packed is None and packed_lm and lm_w is not None:
            V, H = lm_w.shape
            n = ee_lmhead_packed_bytes(V, H)
            if n:
                self.lm_packed = torch.empty(n // 2, dtype=torch.bfloat16, device=dev)
                ee_lmhead_pack_weights(lm_w, self.lm_packed)
                torch.cuda.synchronize(dev)
        self.graph = None

    def _place_tree_kv(self):
        """Set-up for in-place verification (not part of a step): copy node i's
        K/V to cache position ctx + i of its sequence, every layer, and give the
        block table a column for every position below max_ctx + max_T."""
        x = self.inp
        bt, node_off, ctx = x["block_table"], x["node_off"], x["ctx_len"]
        cols = -(-(self.max_ctx + self.max_T) // 16)
        if bt.shape[1] < cols:
            pad = torch.full((self.B, cols - bt.shape[1]), -1, dtype=bt.dtype, device=bt.device)
            x["block_table"] = bt = torch.cat([bt, pad], dim=1).contiguous()
        T = (node_off[1:] - node_off[:-1]).long()
        seq = torch.repeat_interleave(torch.arange(self.B, device=bt.device), T)
        pos = ctx.long()[seq] + (torch.arange(self.total, device=bt.device) - node_off.long()[seq])
        page = bt.long()[seq, pos // 16]
        row = pos % 16
        for name in ("k", "v"):
            cache, tree = x[name + "_cache"], x[name + "_tree"]
            cache[:, page, :, row, :] = tree.permute(1, 0, 2, 3)

    def run(self, stream=None, logits=None, layers=None, marks=None):
        """Enqueue one whole step (``layers`` restricts attention, for tests);
        ``marks(k)`` is called before the first attention layer (k = 0), after
        the last (1) and after the LM head (2), e.g. to record timing events."""
        x = self.inp
        mark = marks if marks is not None else (lambda k: None)
        ee_match_reuse(x["orig_tokens"], x["orig_off"], x["tail"], x["cursor"], self.max_matches,
                       self.match_pos, self.n_matches, self.ws, stream)
        if not self.chain:
            ee_tree_prepare(x["parent"], x["node_off"], self.depth, self.anc, self.ws, stream)
        mark(0)
        for l in (range(self.L) if layers is None else layers):
            out = self.attn_out[l if self.attn_out.shape[0] == self.L else 0]
            if self.chain:
                ee_chain_verify_attn(x["q"][l], x["k_cache"][l], x["v_cache"][l], x["block_table"], x["ctx_len"],
                                     self.max_ctx, x["node_off"], self.max_T, self.scale, out, self.ws, stream)
            elif self.inplace_kv:
                ee_tree_verify_attn_inplace(x["q"][l], x["k_cache"][l], x["v_cache"][l], x["block_table"],
                                            x["ctx_len"], self.max_ctx, x["node_off"], self.anc, self.max_T,
                                            self.scale, out, self.ws, stream)
            else:
                ee_tree_verify_attn(x["q"][l], x["k_tree"][l], x["v_tree"][l], x["k_cache"][l],
                                    x["v_cache"][l], x["block_table"], x["ctx_len"], self.max_ctx,
                                    x["node_off"], self.anc, self.max_T, self.scale, out, self.ws, stream)
        mark(1)
        if self.verify is None and self.lm_packed is not None:
            chain = self.chain
            ee_lmhead_accept_packed(x["hidden"], self.lm_packed, x["lm_w"].shape[0], x["draft_tok"],
                                    None if chain else x["parent"], None if chain else self.depth,
                                    None if chain else self.anc, x["node_off"], self.max_T, self.argmax,
                                    self.accept_len, self.path, self.bonus, self.ws, logits=logits, stream=stream)
        elif self.chain:
            ee_lmhead_accept(x["hidden"], x["lm_w"], x["draft_tok"], None, None, None, x["node_off"], self.max_T,
                             self.argmax, self.accept_len, self.path, self.bonus, self.ws, logits=logits,
                             stream=stream)
        elif self.verify is None:
            ee_lmhead_accept(x["hidden"], x["lm_w"], x["draft_tok"], x["parent"], self.depth, self.anc,
                             x["node_off"], self.max_T, self.argmax, self.accept_len, self.path,
                             self.bonus, self.ws, logits=logits, stream=stream)
        else:
            ee_lmhead_verify(x["hidden"], x["lm_w"], x["draft_tok"], x["parent"], self.depth, self.anc,
                             x["node_off"], self.max_T, self.verify[0], self.verify[1], self.argmax,
                             self.accept_len, self.path, self.bonus, self.ws, gen_mask=self.gen_mask,
                             topk_ids=self.topk_ids, top_tau=self.top_tau, h_norm=self.h_norm,
                             logits=logits, stream=stream)
        mark(2)
        if self.inplace_kv:
            ee_kv_compact_inplace(x["k_cache"], x["v_cache"], x["block_table"], x["ctx_len"], self.ctx_out,
                                  x["node_off"], self.path, self.accept_len, self.total, self.dst_slot,
                                  self.ws, stream)
        else:
            ee_kv_compact(x["k_tree"], x["v_tree"], x["k_cache"], x["v_cache"], x["block_table"],
                          x["ctx_len"], self.ctx_out, x["node_off"], self.path, self.accept_len,
                          self.dst_slot, self.ws, stream)

    def capture(self, stream):
        """Capture one step into a CUDA graph on ``stream`` (a side stream)."""
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            self.run(stream)                       # warm-up outside capture
            stream.synchronize()
            with torch.cuda.graph(g, stream=stream):
                self.run(stream)
        self.graph = g
        return g

    def launches_per_step(self) -> int:
        """Kernels this step launches: match, prepare (not for linear drafts), 1 per attention
        layer, LM head (+ the verification finalize), compaction."""
        return (1 if self.chain else 2) + self.L + 2 + (0 if self.verify is None else 1)


def from_workload(w, device="cuda", keep_layers=True, verify=None, inplace_kv=False, chain=None, packed_lm=True):
    """VerifyStep over a workloads.Workload (its float tensors already on ``device``);
    ``verify`` = (mode, k) uses that rule on the workload's generated branches;
    ``inplace_kv`` verifies with the tree's K/V placed in the cache; ``chain``
    (default: the workload's drafts are all linear and one exceeds 128 tokens)
    verifies linear drafts in place."""
    if chain is None:
        chain = w.max_T > 128
    def i32(a):
        return torch.as_tensor(a, dtype=torch.int32).to(device)
    return VerifyStep(
        orig_tokens=i32(w.orig_tokens), orig_off=torch.as_tensor(w.orig_off, dtype=torch.int64).to(device),
        tail=i32(w.tail), cursor=i32(w.cursor), parent=i32(w.parent), node_off=i32(w.node_off),
        draft_tok=i32(w.draft_tok), ctx_len=i32(w.ctx_len), block_table=i32(w.block_table),
        q=w.q, k_tree=w.k_tree, v_tree=w.v_tree, k_cache=w.k_cache, v_cache=w.v_cache,
        hidden=w.hidden_states, lm_w=w.lm_w, max_ctx=int(w.ctx_len.max()), max_T=w.max_T,
        max_matches=w.max_matches, keep_layers=keep_layers, verify=verify,
        gen_mask=torch.as_tensor(w.gen_mask).to(device) if verify is not None else None,
        inplace_kv=inplace_kv, chain=chain, packed_lm=packed_lm)
