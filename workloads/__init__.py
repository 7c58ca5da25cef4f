"""Seeded synthetic inputs for one edit-oriented verification step.

EfficientEdit (arXiv 2506.02780) measures on CanItEdit and CodeIF-Bench with
Qwen2.5-Coder and DeepSeek-Coder models (Sec. V-A, V-D).  Neither the datasets
nor the weights are used here: these generators stand in for them with random
arrays of the same shapes and reuse structure -- original code ``c`` as a token
array, a generated prefix that copies ``c`` with a few planted edits (Sec. III-A),
a draft tree made of a reuse chain taken from ``c`` plus short generated
branches (gamma = 7-ish, Sec. IV-E), a paged bf16 KV cache, query/hidden states
and LM-head weights.

This module draws random numbers and lays out structure only.  It holds none of
the method's arithmetic: no n-gram matching, attention, projection, argmax or
acceptance is computed here.  Both the fp64 oracle and the CUDA path consume
exactly the arrays produced here.

Integer structure comes from numpy PCG64 (identical on every machine); float
tensors come from a seeded ``torch.Generator`` on the requested device, so the
large configurations can be drawn directly in device memory.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

PAGE = 16            # tokens per KV page
HEAD_DIM = 128
CONFIG_NAMES = ("tiny", "7b", "batched", "33b", "sweep", "long")
BASE_SEED = 1234

# Model shapes of the target models the paper's configurations are named after.
SHAPES = {
    "tiny": dict(n_q=8, n_kv=2, hidden=512, vocab=4096, layers=1),
    "7b": dict(n_q=28, n_kv=4, hidden=3584, vocab=152064, layers=28),
    "33b": dict(n_q=56, n_kv=8, hidden=7168, vocab=32256, layers=62),
}


@dataclass
class TreeSpec:
    """One sequence's draft tree: a reuse chain (root included) plus branches.

    Node numbering: chain nodes 0..chain-1 (node 0 is the root, i.e. the last
    committed token), then each branch's nodes in order.  ``branches`` holds
    (attach_node, length) pairs; a branch's first node is a child of
    ``attach_node``.  ``planted`` is the root-first list of nodes the generator
    wants accepted.
    """
    chain: int
    branches: list
    planted: list = field(default_factory=list)

    @property
    def T(self) -> int:
        return self.chain + sum(b[1] for b in self.branches)

    def parent(self) -> np.ndarray:
        p = [-1] + list(range(self.chain - 1))
        for attach, length in self.branches:
            first = len(p)
            p.append(attach)
            p.extend(range(first, first + length - 1))
        return np.asarray(p, dtype=np.int32)


@dataclass
class Workload:
    name: str
    seed: int
    B: int
    n_q: int
    n_kv: int
    head_dim: int
    hidden: int
    vocab: int
    layers: int
    n: int                       # n-gram length of the reuse match
    max_matches: int
    # reuse match inputs (host numpy)
    orig_tokens: np.ndarray      # int32 [sum len_c]
    orig_off: np.ndarray         # int64 [B+1]
    tail: np.ndarray             # int32 [B, n]
    cursor: np.ndarray           # int32 [B]
    planted_match: np.ndarray    # int32 [B] a position the generator copied the tail from, -1 if none
    # draft tree (host numpy)
    trees: list
    parent: np.ndarray           # int32 [sum T] local parent ids
    node_off: np.ndarray         # int32 [B+1]
    draft_tok: np.ndarray        # int32 [sum T]
    planted_argmax: np.ndarray   # int32 [sum T], -1 where the hidden state is pure noise
    planted_accept: np.ndarray   # int32 [B]
    planted_path: list           # per sequence, root-first local node ids
    # paged KV layout (host numpy)
    ctx_len: np.ndarray          # int32 [B]
    block_table: np.ndarray      # int32 [B, max_pages]
    num_pages: int
    # float tensors (torch, bf16, on `device`)
    q: torch.Tensor              # [L, sum T, n_q, d]
    k_tree: torch.Tensor         # [L, sum T, n_kv, d]
    v_tree: torch.Tensor         # [L, sum T, n_kv, d]
    k_cache: torch.Tensor        # [L, num_pages, n_kv, PAGE, d]
    v_cache: torch.Tensor        # [L, num_pages, n_kv, PAGE, d]
    hidden_states: torch.Tensor  # [sum T, H]
    lm_w: torch.Tensor           # [V, H]
    # edit content: 1 for generated-branch nodes, 0 for the reuse chain (host numpy uint8 [sum T])
    gen_mask: np.ndarray = None

    @property
    def total_nodes(self) -> int:
        return int(self.node_off[-1])

    @property
    def max_T(self) -> int:
        return int(np.diff(self.node_off).max())

    @property
    def max_pages(self) -> int:
        return int(self.block_table.shape[1])

    def seq_tokens(self, s: int) -> np.ndarray:
        return self.orig_tokens[self.orig_off[s]:self.orig_off[s + 1]]


# ----------------------------------------------------------------------------
# original code and generated prefix
# ----------------------------------------------------------------------------

def _original_code(rng, length, vocab, repeat_frac=0.0, seg=8):
    """Uniform tokens; optionally ``repeat_frac`` of them lie in copies of earlier
    ``seg``-token segments (repeated code lines make matches ambiguous).

    The code is cut into ``seg``-token slots; a ``repeat_frac`` share of the
    slots (slot 0 never) are destinations, each overwritten by a copy of an
    earlier ``seg``-token span that starts anywhere but lies wholly inside
    slots that are not destinations.  Copies never land on each other or on a
    source, so every destination is an exact repeat of an earlier span: about
    ``repeat_frac`` of all positions lie in an n-gram (n <= seg) that also
    occurs earlier.  Returns (tokens, list of (src, dst) copy starts, by dst).
    """
    c = rng.integers(0, vocab, size=length, dtype=np.int64).astype(np.int32)
    n_slots = length // seg
    n_seg = min(math.ceil(repeat_frac * length / seg), max(n_slots - 1, 0))
    copies = []
    if n_seg == 0:
        return c, copies
    dst_slots = np.sort(rng.choice(np.arange(1, n_slots), size=n_seg, replace=False))
    is_dst = np.zeros(n_slots + 1, dtype=bool)
    is_dst[dst_slots] = True
    for ds in dst_slots:
        dst = int(ds) * seg
        for _ in range(64):      # a span starting anywhere before dst, clear of destinations
            src = int(rng.integers(0, dst - seg + 1))
            if not (is_dst[src // seg] or is_dst[(src + seg - 1) // seg]):
                break
        else:
            continue             # no clear span found (rare, early slots): no copy
        c[dst:dst + seg] = c[src:src + seg]
        copies.append((src, dst))
    return c, copies


def _prefix_with_edits(rng, c, plen, n_edits, vocab, edit_len=8, keep_tail=4):
    """Generated prefix = c[:plen] with ``n_edits`` random ``edit_len``-token edits
    planted before the last ``keep_tail`` tokens.  Returns (prefix, last_edit_end)."""
    prefix = c[:plen].copy()
    last_end = 0
    hi = plen - keep_tail - edit_len
    if n_edits and hi > 0:
        starts = np.sort(rng.choice(np.arange(0, hi + 1), size=min(n_edits, hi + 1), replace=False))
        for s0 in starts:
            prefix[s0:s0 + edit_len] = rng.integers(0, vocab, size=edit_len)
            last_end = max(last_end, int(s0) + edit_len)
    return prefix, last_end


# ----------------------------------------------------------------------------
# trees and planted targets
# ----------------------------------------------------------------------------

def _distinct_token(rng, vocab, avoid):
    while True:
        t = int(rng.integers(0, vocab))
        if t not in avoid:
            return t


def _tree_tokens(rng, spec, chain_tokens, vocab):
    """Chain nodes carry ``chain_tokens``; branch tokens are random and differ
    from their siblings' tokens."""
    parent = spec.parent()
    tok = np.empty(spec.T, dtype=np.int32)
    tok[:spec.chain] = chain_tokens[:spec.chain]
    for i in range(spec.chain, spec.T):
        sib = {int(tok[j]) for j in range(i) if parent[j] == parent[i]}
        tok[i] = _distinct_token(rng, vocab, sib)
    return tok


def _planted_targets(rng, spec, tok, vocab, noise_frac):
    """Token the generator wants argmax(node) to be.  Along the planted path each
    node targets its successor's token; the path's last node targets a token no
    child carries; other nodes get a random target or none (-1, pure noise)."""
    parent = spec.parent()
    children = [[] for _ in range(spec.T)]
    for i in range(1, spec.T):
        children[parent[i]].append(i)
    tgt = np.full(spec.T, -1, dtype=np.int32)
    path = spec.planted
    on_path = set(path)
    for a, b in zip(path[:-1], path[1:]):
        tgt[a] = tok[b]
    last = path[-1]
    tgt[last] = _distinct_token(rng, vocab, {int(tok[c]) for c in children[last]})
    for u in range(spec.T):
        if u in on_path:
            continue
        if rng.random() < noise_frac:
            continue
        tgt[u] = _distinct_token(rng, vocab, {int(tok[c]) for c in children[u]})
    return tgt


def chain_path(depth):
    return list(range(depth + 1))


# ----------------------------------------------------------------------------
# per-configuration sequence plans
# ----------------------------------------------------------------------------

def _plan(name, rng, overrides):
    """Return (shape dict, per-sequence list of dicts with len_c, ctx, spec, prefix params)."""
    o = dict(overrides)
    if name == "tiny":
        shape = dict(SHAPES["tiny"], n=4)
        seqs = [dict(len_c=400, ctx=512, plen=300, edits=3,
                     spec=TreeSpec(12, [(0, 4)], chain_path(7)))]
    elif name == "7b":
        shape = dict(SHAPES["7b"], n=4)
        seqs = [dict(len_c=3000, ctx=4096, plen=2000, edits=3,
                     spec=TreeSpec(48, [(0, 8), (24, 8)], chain_path(30)))]
    elif name == "33b":
        shape = dict(SHAPES["33b"], n=4)
        attach = sorted(int(a) for a in rng.choice(np.arange(0, 100), size=4, replace=False))
        seqs = [dict(len_c=28000, ctx=32768, plen=20000, edits=20,
                     spec=TreeSpec(112, [(a, 4) for a in attach], chain_path(100)))]
    elif name == "batched":
        shape = dict(SHAPES["7b"], n=4)
        seqs = []
        for _ in range(8):
            ctx = int(rng.integers(1024, 16385))
            T = int(rng.integers(32, 97))
            frac = float(rng.uniform(0.5, 0.9))
            chain = max(2, min(T - 2, int(round(frac * T))))
            rest = T - chain
            b1 = rest // 2
            b2 = rest - b1
            at2 = int(rng.integers(1, chain))
            branches = [(0, b1), (at2, b2)] if b1 > 0 else [(at2, b2)]
            spec = TreeSpec(chain, branches)
            if rng.random() < 0.3:
                # accepted path leaves the reuse chain into the second branch
                first = chain + (b1 if b1 > 0 else 0)
                depth_in = int(rng.integers(1, b2 + 1))
                spec.planted = chain_path(at2) + list(range(first, first + depth_in))
            else:
                spec.planted = chain_path(int(rng.integers(1, chain)))
            len_c = int(round(0.8 * ctx))
            seqs.append(dict(len_c=len_c, ctx=ctx, plen=int(0.6 * len_c), edits=3, spec=spec))
    elif name == "long":
        # a long reuse draft verified in one pass (Sec. III-A: a reused span of
        # the original code needs no draft length): 7B shapes, one sequence, a
        # 2048-token chain of the original code after the match point, accepted
        # up to an edit 1500 tokens in
        shape = dict(SHAPES["7b"], n=4)
        seqs = [dict(len_c=8000, ctx=4096, plen=3000, edits=3,
                     spec=TreeSpec(2048, [], chain_path(1500)))]
    elif name == "sweep":
        shape = dict(SHAPES["7b"], n=o.pop("n", 4))
        seqs = []
        for _ in range(o.pop("B", 32)):
            plen_nodes = int(rng.integers(1, 129))
            spec = TreeSpec(128, [], chain_path(plen_nodes - 1))
            seqs.append(dict(len_c=65536, ctx=int(rng.integers(0, 1025)), plen=None, edits=0,
                             spec=spec))
    else:
        raise ValueError(f"unknown configuration {name!r}")
    for key in ("n_q", "n_kv", "hidden", "vocab", "layers", "n"):
        if key in o:
            shape[key] = o.pop(key)
    if "ctx" in o:
        c = o.pop("ctx")
        for s in seqs:
            s["ctx"] = int(c)
    if "trees" in o:
        specs = o.pop("trees")
        seqs = [dict(seqs[i % len(seqs)], spec=sp) for i, sp in enumerate(specs)]
    if "ctxs" in o:
        # one context length per sequence (after ``trees`` fixed the count)
        cs = [int(c) for c in o.pop("ctxs")]
        if len(cs) != len(seqs):
            raise ValueError("ctxs needs one entry per sequence")
        seqs = [dict(sp, ctx=c) for sp, c in zip(seqs, cs)]
    if o:
        raise ValueError(f"unused overrides {sorted(o)}")
    return shape, seqs


# ----------------------------------------------------------------------------
# float tensors
# ----------------------------------------------------------------------------

def _randn_bf16(gen, shape, std, device, chunk_rows=None):
    out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    flat = out.view(shape[0], -1)
    step = chunk_rows or shape[0]
    for r0 in range(0, shape[0], step):
        r1 = min(shape[0], r0 + step)
        t = torch.randn((r1 - r0, flat.shape[1]), generator=gen, device=device, dtype=torch.float32)
        flat[r0:r1] = (t * std).to(torch.bfloat16)
    return out


def _lm_inputs(gen, rng, V, H, total, planted_argmax, draft_tok, dup_rows, plant_scale, device,
               extra=None):
    """LM-head weight W ~ N(0, 0.02^2) and hidden states.  A planted node's hidden
    state is plant_scale * (unit vector along W[target]) + N(0, 1) noise, so its
    target wins by a wide logit margin; other nodes get pure noise.  ``extra``
    maps a node to (tokens, logits): its hidden state is then replaced by the
    least-squares vector h = W_P^T (W_P W_P^T)^-1 L that gives exactly those
    logits to those tokens (W_P their rows), plus N(0, 0.05^2) noise -- ranked
    planting with controlled gaps."""
    lm_w = _randn_bf16(gen, (V, H), 0.02, device, chunk_rows=16384)
    if dup_rows:
        # exact ties: a planted target row is copied to a higher, unused token id
        used = {int(t) for t in planted_argmax if t >= 0} | {int(x) for x in draft_tok}
        n_dup = 0
        for t in sorted({int(t) for t in planted_argmax if 0 <= t < V - 1}):
            if n_dup == dup_rows:
                break
            hi = int(rng.integers(t + 1, V))
            if hi in used:
                continue
            lm_w[hi] = lm_w[t]
            used.add(hi)
            n_dup += 1
    hidden = torch.randn((total, H), generator=gen, device=device, dtype=torch.float32)
    idx = np.nonzero(planted_argmax >= 0)[0]
    if len(idx):
        rows = lm_w[torch.as_tensor(planted_argmax[idx], device=device, dtype=torch.long)].float()
        unit = rows / rows.norm(dim=1, keepdim=True)
        sel = torch.as_tensor(idx, device=device, dtype=torch.long)
        hidden[sel] = hidden[sel] + plant_scale * unit
    for node, (toks, lgts) in sorted((extra or {}).items()):
        wp = lm_w[torch.as_tensor(toks, device=device, dtype=torch.long)].double()
        lv = torch.as_tensor(lgts, device=device, dtype=torch.float64)
        h = wp.T @ torch.linalg.solve(wp @ wp.T, lv)
        hidden[node] = h.float() + 0.05 * torch.randn(H, generator=gen, device=device)
    return lm_w, hidden.to(torch.bfloat16)


def build(name: str, seed: int | None = None, device="cpu", *, q_std: float = 1.0,
          plant_scale: float = 12.0, noise_frac: float = 0.1, max_matches: int = 8,
          dup_rows: int = 0, lm_head: bool | None = None, verify_plant: bool = False,
          **overrides) -> Workload:
    """Draw one workload.

    ``name`` is one of CONFIG_NAMES; ``seed`` defaults to 1234 + the config's
    index.  Overrides (``ctx``, ``layers``, ``vocab``, ``hidden``, ``n_q``,
    ``n_kv``, ``n``, ``trees``, ``ctxs`` (one context length per sequence), and
    for the sweep ``B``) shrink or reshape a
    configuration for tests.  ``q_std`` scales the queries (a large value makes
    the softmax peaky).  ``dup_rows`` > 0 copies that many planted target rows of
    the LM-head weight to a higher token id, creating exact logit ties.
    ``lm_head`` (default: every configuration but the sweep) draws the LM-head
    weight and hidden states; without it both are None.  ``verify_plant`` puts
    the draft token of every generated node on a planted path at rank 0, 1 or 2
    of its parent's distribution, between decoy tokens: exact logits top, top -
    gap, top - 2 gap, ... with top = ln(V) + 8 and gap 0.1, 0.6 or 3.0 (so the
    entropy-aware rule meets near-uniform, medium and peaked positions);
    planted_accept / planted_path then describe the greedy rule only up to the
    first edge planted below rank 0.
    """
    if seed is None:
        seed = BASE_SEED + CONFIG_NAMES.index(name)
    rng = np.random.Generator(np.random.PCG64(seed))
    shape, seqs = _plan(name, rng, overrides)
    n, V = shape["n"], shape["vocab"]
    B = len(seqs)

    # --- original code, prefix tail, cursor, reuse chain -------------------
    codes, tails, cursors, planted_match, chain_toks = [], [], [], [], []
    for sp in seqs:
        rep = 0.3 if name == "sweep" else 0.0
        c, copies = _original_code(rng, sp["len_c"], V, repeat_frac=rep)
        chain = sp["spec"].chain
        if sp["plen"] is None:
            # sweep: tail copied from a random location (90%) or random (10%)
            cur = int(rng.integers(0, len(c) // 2))
            u = rng.random()
            late = [(a, b) for a, b in copies[-64:] if a >= cur and b + n < len(c)]
            if u < 0.3 and late and n <= 8:
                # tail taken from a repeated segment: it matches at least twice
                a, b = late[int(rng.integers(0, len(late)))]
                tail = c[b:b + n].copy()
                pm = b
            elif u < 0.9:
                p = int(rng.integers(cur, len(c) - n))
                tail = c[p:p + n].copy()
                pm = p
            else:
                tail = rng.integers(0, V, size=n).astype(np.int32)
                pm = -1
            ct = rng.integers(0, V, size=chain).astype(np.int32)
        else:
            plen = min(sp["plen"], len(c) - chain - 1)
            prefix, last_end = _prefix_with_edits(rng, c, plen, sp["edits"], V, keep_tail=n)
            tail = prefix[plen - n:plen].copy()
            pm = plen - n
            cur = min(last_end, pm)
            # reuse chain: root = last matched token c[p+n-1], drafts follow it in c
            ct = c[pm + n - 1: pm + n - 1 + chain].copy()
        codes.append(c)
        tails.append(tail)
        cursors.append(cur)
        planted_match.append(pm)
        chain_toks.append(ct)
    orig_off = np.zeros(B + 1, dtype=np.int64)
    orig_off[1:] = np.cumsum([len(c) for c in codes])
    orig_tokens = np.concatenate(codes).astype(np.int32)

    # --- draft trees and planted targets ------------------------------------
    parents, toks, tgts, paths = [], [], [], []
    for sp, ct in zip(seqs, chain_toks):
        spec = sp["spec"]
        if not spec.planted:
            spec.planted = [0]
        tok = _tree_tokens(rng, spec, ct, V)
        parents.append(spec.parent())
        toks.append(tok)
        tgts.append(_planted_targets(rng, spec, tok, V, noise_frac))
        paths.append(list(spec.planted))
    node_off = np.zeros(B + 1, dtype=np.int32)
    node_off[1:] = np.cumsum([len(p) for p in parents])
    parent = np.concatenate(parents).astype(np.int32)
    draft_tok = np.concatenate(toks).astype(np.int32)
    planted_argmax = np.concatenate(tgts).astype(np.int32)
    planted_accept = np.asarray([len(p) - 1 for p in paths], dtype=np.int32)
    total = int(node_off[-1])
    gen_mask = np.concatenate([(np.arange(sp["spec"].T) >= sp["spec"].chain) for sp in seqs]
                              ).astype(np.uint8)
    extra = {}
    if verify_plant:
        # ranked planting on generated edges of the planted paths: the draft token
        # gets rank r; decoys fill the other ranks down to r + 2, scales falling by
        # `gap` per rank
        for s_i, (sp, pth) in enumerate(zip(seqs, paths)):
            o = int(node_off[s_i])
            for a, b in zip(pth[:-1], pth[1:]):
                if not gen_mask[o + b]:
                    continue
                r = int(rng.integers(0, 3))
                gap = float(rng.choice([0.1, 0.6, 3.0]))
                avoid = {int(draft_tok[o + b])} | {int(x) for x in draft_tok[o:o + sp["spec"].T]}
                ranked = []
                for j in range(r + 3):
                    if j == r:
                        ranked.append(int(draft_tok[o + b]))
                    else:
                        t = _distinct_token(rng, V, avoid)
                        avoid.add(t)
                        ranked.append(t)
                planted_argmax[o + a] = ranked[0]
                top = math.log(V) + 8.0
                extra[o + a] = (ranked, [top - gap * j for j in range(len(ranked))])

    # --- paged KV layout: ctx + T slots per sequence, random page order -----
    ctx_len = np.asarray([sp["ctx"] for sp in seqs], dtype=np.int32)
    Ts = np.diff(node_off)
    pages_per = [max(1, math.ceil((int(c) + int(t)) / PAGE)) for c, t in zip(ctx_len, Ts)]
    num_pages = int(sum(pages_per))
    perm = rng.permutation(num_pages).astype(np.int32)
    max_pages = max(pages_per)
    block_table = np.full((B, max_pages), -1, dtype=np.int32)
    o = 0
    for s, npg in enumerate(pages_per):
        block_table[s, :npg] = perm[o:o + npg]
        o += npg

    # --- float tensors -------------------------------------------------------
    L, n_q, n_kv, H = shape["layers"], shape["n_q"], shape["n_kv"], shape["hidden"]
    d = HEAD_DIM
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    kv_std = 1.0 / math.sqrt(d)
    q = _randn_bf16(gen, (L, total, n_q, d), q_std, device)
    k_tree = _randn_bf16(gen, (L, total, n_kv, d), kv_std, device)
    v_tree = _randn_bf16(gen, (L, total, n_kv, d), kv_std, device)
    k_cache = _randn_bf16(gen, (L, num_pages, n_kv, PAGE, d), kv_std, device, chunk_rows=1)
    v_cache = _randn_bf16(gen, (L, num_pages, n_kv, PAGE, d), kv_std, device, chunk_rows=1)
    if lm_head is None:
        lm_head = name != "sweep"
    lm_w = hidden_states = None
    if lm_head:
        lm_w, hidden_states = _lm_inputs(gen, rng, V, H, total, planted_argmax, draft_tok,
                                         dup_rows, plant_scale, device, extra)

    return Workload(

        name=name, seed=seed, B=B, n_q=n_q, n_kv=n_kv, head_dim=d, hidden=H, vocab=V, layers=L,
        n=n, max_matches=max_matches,
        orig_tokens=orig_tokens, orig_off=orig_off, tail=np.stack(tails).astype(np.int32),
        cursor=np.asarray(cursors, dtype=np.int32), planted_match=np.asarray(planted_match, dtype=np.int32),
        trees=[sp["spec"] for sp in seqs], parent=parent, node_off=node_off, draft_tok=draft_tok,
        planted_argmax=planted_argmax, planted_accept=planted_accept, planted_path=paths,
        ctx_len=ctx_len, block_table=block_table, num_pages=num_pages,
        q=q, k_tree=k_tree, v_tree=v_tree, k_cache=k_cache, v_cache=v_cache,
        hidden_states=hidden_states, lm_w=lm_w, gen_mask=gen_mask,
    )


def describe(w: Workload) -> dict:
    """Short description of a workload for JSON output."""
    Ts = np.diff(w.node_off)
    return {
        "workload": w.name, "B": w.B, "ctx": [int(c) for c in w.ctx_len][:8],
        "T": [int(t) for t in Ts][:8], "n_q": w.n_q, "n_kv": w.n_kv, "head_dim": w.head_dim,
        "hidden": w.hidden, "vocab": w.vocab, "layers": w.layers, "n_gram": w.n,
        "page": PAGE, "seed": w.seed,
    }
