"""fp64 CPU oracle for the EfficientEdit verification step (test infrastructure).

Only tests, ``__graft_entry__.smoke()`` and bench.py's CPU-baseline leg use this
module.  Each function cites the passage of EfficientEdit (arXiv 2506.02780) it
follows and states the reading taken where the paper is silent.

Notation: B sequences; sequence s owns tree nodes node_off[s]..node_off[s+1]-1
(local ids 0..T_s-1, local 0 is the root = last committed token); ctx = cached
context length; the KV cache is paged, PAGE tokens per page, laid out
[num_pages, n_kv, PAGE, d]; query head h reads KV head h // (n_q / n_kv).
"""
from __future__ import annotations

import math

import numpy as np

PAGE = 16
_U32 = 2.0 ** -24          # unit roundoff of fp32


def _raw16(t):
    """Raw 16-bit patterns of a bf16 torch tensor as a numpy uint16 array (for copies)."""
    import torch
    return t.detach().to("cpu").contiguous().view(torch.int16).numpy().view(np.uint16)


def _f64(x):
    """Exact fp64 copy of a bf16/fp32 tensor or array."""
    if hasattr(x, "detach"):
        return x.detach().to("cpu").double().numpy()
    return np.asarray(x, dtype=np.float64)


# ----------------------------------------------------------------------------
# (1) reuse-span match -- Sec. III-A, prefix matching to switch back to Reuse
# ----------------------------------------------------------------------------

def match_reuse(orig_tokens, orig_off, tail, cursor, max_matches):
    """Positions p in the remaining original code where the last n generated
    tokens occur: c[p:p+n] == tail, searched from the cursor onwards.

    Sec. III-A: when Generate switches back to Reuse, positions of the remaining
    ``c`` that match the suffix of what was generated become new draft starts;
    the tokens of ``c`` after such a position are the reuse draft.
    Readings: every position p >= cursor is searched (not only p == cursor);
    a match must leave at least one draft token, p + n < len(c); several match
    points are returned in ascending order, up to ``max_matches``, with the
    total count.

    Returns (match_pos int32 [B, max_matches] padded with -1, n_matches int32 [B]).
    """
    orig_tokens = np.asarray(orig_tokens)
    orig_off = np.asarray(orig_off)
    tail = np.asarray(tail)
    cursor = np.asarray(cursor)
    B, n = tail.shape
    if n < 1:
        raise ValueError("n must be >= 1")
    if max_matches < 1:
        raise ValueError("max_matches must be >= 1")
    match_pos = np.full((B, max_matches), -1, dtype=np.int32)
    n_matches = np.zeros(B, dtype=np.int32)
    for s in range(B):
        c = orig_tokens[orig_off[s]:orig_off[s + 1]]
        if cursor[s] < 0:
            raise ValueError("cursor must be >= 0")
        if len(c) < n + 1:
            continue
        windows = np.lib.stride_tricks.sliding_window_view(c, n)   # windows[p] = c[p:p+n]
        hit = np.all(windows == tail[s][None, :], axis=1)
        pos = np.nonzero(hit)[0]
        pos = pos[(pos >= cursor[s]) & (pos + n < len(c))]
        n_matches[s] = len(pos)
        k = min(len(pos), max_matches)
        match_pos[s, :k] = pos[:k]
    return match_pos, n_matches


# ----------------------------------------------------------------------------
# (2) draft-tree structure
# ----------------------------------------------------------------------------

def tree_prepare(parent, node_off, max_nodes=128):
    """depth and ancestor set of every draft-tree node.

    The paper's drafts are linear (Sec. III-A); a tree generalises them to
    several drafts sharing a prefix (several match points, Sec. III-A, plus
    generated branches).  depth(root) = 0, depth(i) = depth(parent(i)) + 1;
    anc(i) = anc(parent(i)) U {i}.  Parents precede children (parent[i] < i).

    Returns (depth int32 [sum T], anc uint64 [sum T, 2]) where bit j of
    anc[i] (word j // 64) is set when local node j is on the root-to-i path.
    """
    parent = np.asarray(parent)
    node_off = np.asarray(node_off)
    total = int(node_off[-1])
    depth = np.zeros(total, dtype=np.int32)
    anc = np.zeros((total, 2), dtype=np.uint64)
    for s in range(len(node_off) - 1):
        o, T = int(node_off[s]), int(node_off[s + 1] - node_off[s])
        if T < 1 or T > max_nodes:
            raise ValueError("each tree needs 1..%d nodes" % max_nodes)
        sets = []
        for i in range(T):
            p = int(parent[o + i])
            if i == 0:
                if p != -1:
                    raise ValueError("node 0 must be the root (parent -1)")
                depth[o] = 0
                sets.append({0})
            else:
                if not (0 <= p < i):
                    raise ValueError("parent[i] must satisfy 0 <= parent[i] < i")
                depth[o + i] = depth[o + p] + 1
                sets.append(sets[p] | {i})
            for j in sets[i]:
                anc[o + i, j // 64] |= np.uint64(1) << np.uint64(j % 64)
    return depth, anc


def anc_to_sets(anc_row):
    """Set of local node ids encoded in one [2] uint64 ancestor row."""
    out = set()
    for w in range(2):
        v = int(anc_row[w])
        for b in range(64):
            if (v >> b) & 1:
                out.add(64 * w + b)
    return out


# ----------------------------------------------------------------------------
# (3) tree-masked attention over the paged cache -- Sec. III-A, one target pass
# ----------------------------------------------------------------------------

def _context_kv(cache_l, block_table_row, ctx, hk):
    """[ctx, d] fp64 rows of one KV head for cached positions 0..ctx-1."""
    if ctx == 0:
        return np.zeros((0, cache_l.shape[-1]))
    npg = (ctx + PAGE - 1) // PAGE
    pages = np.asarray(block_table_row[:npg])
    if np.any(pages < 0) or np.any(pages >= cache_l.shape[0]):
        raise ValueError("block table entry out of range")
    rows = cache_l[pages, hk]                     # [npg, PAGE, d]
    return rows.reshape(npg * PAGE, -1)[:ctx]


def tree_attention(q, k_tree, v_tree, k_cache, v_cache, block_table, ctx_len, node_off, anc,
                   scale=None, nodes=None, heads=None):
    """Attention output of every draft node for ONE layer.

    Sec. III-A: one forward pass of the target over (prefix, draft) scores every
    draft token.  With a tree, node i attends to the cached prefix (positions
    0..ctx-1, read through the block table) and to the tree nodes on its own
    root-to-i path (its ancestor set, i included) -- exactly what it would see
    if its path were appended to the prefix as a linear draft.

    o[i, h] = sum_j softmax_j(scale * q[i, h] . k_j) v_j, j over those keys,
    with k_j, v_j from KV head h // (n_q / n_kv).  scale defaults to 1/sqrt(d).
    Inputs are one layer: q [sumT, n_q, d], k_tree/v_tree [sumT, n_kv, d],
    k_cache/v_cache [num_pages, n_kv, PAGE, d].

    ``nodes`` (global node ids) and ``heads`` restrict the computation to a
    sample; other entries of the returned fp64 [sumT, n_q, d] array are NaN.
    """
    q = _f64(q)
    kt, vt = _f64(k_tree), _f64(v_tree)
    kc, vc = _f64(k_cache), _f64(v_cache)
    total, n_q, d = q.shape
    n_kv = kt.shape[1]
    if n_q % n_kv:
        raise ValueError("n_q must be a multiple of n_kv")
    g = n_q // n_kv
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    node_off = np.asarray(node_off)
    want_nodes = set(range(total)) if nodes is None else set(int(x) for x in nodes)
    want_heads = list(range(n_q)) if heads is None else [int(h) for h in heads]
    out = np.full((total, n_q, d), np.nan)
    for s in range(len(node_off) - 1):
        o, T = int(node_off[s]), int(node_off[s + 1] - node_off[s])
        ctx = int(ctx_len[s])
        for hk in range(n_kv):
            hs = [h for h in want_heads if h // g == hk]
            if not hs:
                continue
            kctx = _context_kv(kc, block_table[s], ctx, hk)
            vctx = _context_kv(vc, block_table[s], ctx, hk)
            for i in range(T):
                if o + i not in want_nodes:
                    continue
                path = sorted(anc_to_sets(anc[o + i]))
                if any(j >= T for j in path):
                    raise ValueError("ancestor outside the tree")
                keys = np.concatenate([kctx, kt[[o + j for j in path], hk]], axis=0)
                vals = np.concatenate([vctx, vt[[o + j for j in path], hk]], axis=0)
                for h in hs:
                    sc = scale * (keys @ q[o + i, h])
                    p = np.exp(sc - sc.max())
                    p /= p.sum()
                    out[o + i, h] = p @ vals
    return out


# ----------------------------------------------------------------------------
# (4) LM head, decode() = argmax, greedy acceptance -- Eq. (piecewise)
# ----------------------------------------------------------------------------

def lm_head_logits(hidden, lm_w, rows=None):
    """logits[i, v] = hidden[i] . W[v] in fp64 (W is [V, H], vocab-major), and
    the fp32 accumulation bound err[i, v] = 2 H 2^-24 sum_k |hidden[i,k] W[v,k]|
    that separates honest near-ties from wrong answers.  ``rows`` restricts the
    vocabulary to a slice (for bounded CPU timing)."""
    x = _f64(hidden)
    w = _f64(lm_w if rows is None else lm_w[rows])
    logits = x @ w.T
    err = 2.0 * x.shape[1] * _U32 * (np.abs(x) @ np.abs(w).T)
    return logits, err


def lm_head_argmax(hidden, lm_w):
    """decode(p_i) of Eq. (piecewise): greedy decoding, the token of highest
    probability, i.e. the argmax of the logits.  Ties go to the lowest token id.

    Returns (argmax int32 [sumT], candidates list of int arrays, logits fp64).
    ``candidates[i]`` holds every token whose logit is within the fp32
    accumulation bound of the maximum -- any fp32 implementation may return one
    of them; when it has one element the answer is unique.
    """
    logits, err = lm_head_logits(hidden, lm_w)
    am = np.argmax(logits, axis=1).astype(np.int32)   # first occurrence = lowest id
    cands = []
    for i in range(logits.shape[0]):
        lo = np.max(logits[i] - err[i])
        cands.append(np.nonzero(logits[i] + err[i] >= lo)[0].astype(np.int32))
    return am, cands, logits


def accept_path(argmax, draft_tok, parent, node_off, max_T=None):
    """Longest accepted draft path per sequence -- Eq. (piecewise).

    In a linear draft the logits at d_{i-1} (the root for i = 1) give p_i, and
    d_1..d_j are accepted for the largest j with decode(p_i) = d_i for all
    i <= j.  In a tree, node u is accepted when every edge (a -> b) on its
    root-to-u path has draft_tok[b] == argmax[a].  The accepted path is the
    deepest accepted node's root-to-node path; among equally deep nodes the
    lowest node id wins (this only matters when siblings carry equal tokens).
    accept_len = that node's depth (drafts accepted, root excluded); bonus =
    argmax at that node, the target's own next token (Sec. II-B: the token
    sampled from the last distribution is kept as well).

    Returns (accept_len int32 [B], path int32 [B, max_T] root-first local ids
    padded with -1, bonus int32 [B]).
    """
    argmax = np.asarray(argmax)
    draft_tok = np.asarray(draft_tok)
    parent = np.asarray(parent)
    node_off = np.asarray(node_off)
    B = len(node_off) - 1
    Ts = np.diff(node_off)
    if max_T is None:
        max_T = int(Ts.max())
    accept_len = np.zeros(B, dtype=np.int32)
    path = np.full((B, max_T), -1, dtype=np.int32)
    bonus = np.zeros(B, dtype=np.int32)
    for s in range(B):
        o, T = int(node_off[s]), int(Ts[s])
        accepted = [False] * T
        depth = [0] * T
        accepted[0] = True
        for i in range(1, T):
            p = int(parent[o + i])
            depth[i] = depth[p] + 1
            accepted[i] = accepted[p] and int(draft_tok[o + i]) == int(argmax[o + p])
        best = 0
        for i in range(1, T):
            if accepted[i] and depth[i] > depth[best]:
                best = i
        chain = []
        u = best
        while u != -1:
            chain.append(u)
            u = int(parent[o + u]) if u != 0 else -1
        chain.reverse()
        accept_len[s] = depth[best]
        path[s, :len(chain)] = chain
        bonus[s] = int(argmax[o + best])
    return accept_len, path, bonus


# ----------------------------------------------------------------------------
# (5) KV compaction of the accepted path -- Sec. III-A, accepted tokens extend prefix
# ----------------------------------------------------------------------------

def kv_compact(k_tree, v_tree, k_cache, v_cache, block_table, ctx_len, node_off, path, accept_len):
    """Append the accepted path's K/V to the paged cache, every layer.

    Sec. III-A: accepted draft tokens extend the prefix; their keys/values were
    computed in the verification pass, so they become cache entries.  Path entry
    k (k = 0..accept_len, the root first) goes to position ctx + k, i.e. slot
    block_table[(ctx+k) // PAGE] * PAGE + (ctx+k) % PAGE.  The bonus token's K/V
    is not computed in this pass; it becomes the next root.

    k_tree/v_tree: [L, sumT, n_kv, d]; k_cache/v_cache: [L, num_pages, n_kv,
    PAGE, d] (numpy, any dtype; copies are returned).
    Returns (k_cache', v_cache', dst_slot int32 [B, max_T] padded with -1,
    ctx_len' int32 [B] = ctx + accept_len + 1).
    """
    kc = np.array(k_cache, copy=True)
    vc = np.array(v_cache, copy=True)
    kt, vt = np.asarray(k_tree), np.asarray(v_tree)
    node_off = np.asarray(node_off)
    B = len(node_off) - 1
    max_T = path.shape[1]
    dst = np.full((B, max_T), -1, dtype=np.int32)
    ctx_out = np.asarray(ctx_len, dtype=np.int32).copy()
    for s in range(B):
        ctx = int(ctx_len[s])
        for k in range(int(accept_len[s]) + 1):
            node = int(path[s, k])
            pos = ctx + k
            page = int(block_table[s, pos // PAGE])
            if page < 0 or page >= kc.shape[1]:
                raise ValueError("no page allocated for position %d" % pos)
            off = pos % PAGE
            dst[s, k] = page * PAGE + off
            src = int(node_off[s]) + node
            kc[:, page, :, off, :] = kt[:, src, :, :]
            vc[:, page, :, off, :] = vt[:, src, :, :]
        ctx_out[s] = ctx + int(accept_len[s]) + 1
    return kc, vc, dst, ctx_out


# ----------------------------------------------------------------------------
# In-place speculative K/V: the tree's K/V live in the cache slots after the
# context (the accepted prefix extension of Sec. III-A without a separate
# tree buffer)
# ----------------------------------------------------------------------------

def _slot(block_table, s, pos, num_pages):
    page = int(block_table[s, pos // PAGE])
    if page < 0 or page >= num_pages:
        raise ValueError("no page allocated for position %d" % pos)
    return page, pos % PAGE


def tree_kv_to_cache(k_tree, v_tree, k_cache, v_cache, block_table, ctx_len, node_off):
    """Place every tree node's K/V at cache position ctx + i (i = its local id),
    every layer: where a K/V projection writes them when the tree is verified in
    place.  Shapes as in kv_compact; copies are returned."""
    kc = np.array(k_cache, copy=True)
    vc = np.array(v_cache, copy=True)
    kt, vt = np.asarray(k_tree), np.asarray(v_tree)
    node_off = np.asarray(node_off)
    for s in range(len(node_off) - 1):
        o, T, ctx = int(node_off[s]), int(node_off[s + 1] - node_off[s]), int(ctx_len[s])
        for i in range(T):
            page, off = _slot(block_table, s, ctx + i, kc.shape[1])
            kc[:, page, :, off, :] = kt[:, o + i, :, :]
            vc[:, page, :, off, :] = vt[:, o + i, :, :]
    return kc, vc


def tree_kv_from_cache(k_cache, v_cache, block_table, ctx_len, node_off, n_layers=None):
    """The tree's K/V as a [L, sumT, n_kv, d] array, read from positions ctx + i:
    what attention over an in-place tree sees as the tree keys."""
    kc, vc = np.asarray(k_cache), np.asarray(v_cache)
    node_off = np.asarray(node_off)
    L = kc.shape[0] if n_layers is None else n_layers
    total = int(node_off[-1])
    kt = np.zeros((L, total) + kc.shape[2:3] + kc.shape[4:], dtype=kc.dtype)
    vt = np.zeros_like(kt)
    for s in range(len(node_off) - 1):
        o, T, ctx = int(node_off[s]), int(node_off[s + 1] - node_off[s]), int(ctx_len[s])
        for i in range(T):
            page, off = _slot(block_table, s, ctx + i, kc.shape[1])
            kt[:, o + i] = kc[:L, page, :, off, :]
            vt[:, o + i] = vc[:L, page, :, off, :]
    return kt, vt


def kv_compact_inplace(k_cache, v_cache, block_table, ctx_len, node_off, path, accept_len):
    """Compaction when the tree's K/V already sit at positions ctx + i.

    The accepted path (root first) must end up at positions ctx .. ctx + acc,
    as kv_compact appends it.  Path entry k is node path[k] >= k (a parent's id
    is below its child's), already at ctx + path[k]: entries with path[k] == k
    stay, the others move down to ctx + k.  Moving in increasing k reads every
    source before a later move overwrites it (a source ctx + path[k] is above
    every earlier destination and at most the destination of a later entry
    k' > k with path[k] == k').  Returns (k_cache', v_cache', dst_slot int32
    [B, max_T] padded with -1, ctx_len' int32 [B] = ctx + accept_len + 1).
    """
    kc = np.array(k_cache, copy=True)
    vc = np.array(v_cache, copy=True)
    node_off = np.asarray(node_off)
    B = len(node_off) - 1
    max_T = path.shape[1]
    dst = np.full((B, max_T), -1, dtype=np.int32)
    ctx_out = np.asarray(ctx_len, dtype=np.int32).copy()
    for s in range(B):
        ctx = int(ctx_len[s])
        for k in range(int(accept_len[s]) + 1):
            node = int(path[s, k])
            dpage, doff = _slot(block_table, s, ctx + k, kc.shape[1])
            dst[s, k] = dpage * PAGE + doff
            if node != k:
                spage, soff = _slot(block_table, s, ctx + node, kc.shape[1])
                kc[:, dpage, :, doff, :] = kc[:, spage, :, soff, :]
                vc[:, dpage, :, doff, :] = vc[:, spage, :, soff, :]
        ctx_out[s] = ctx + int(accept_len[s]) + 1
    return kc, vc, dst, ctx_out


# ----------------------------------------------------------------------------
# Long reuse drafts: a linear draft of up to 2048 tokens verified in place
# (Sec. III-A: the reused span of the original code needs no draft length)
# ----------------------------------------------------------------------------

def chain_attention(q, k_cache, v_cache, block_table, ctx_len, node_off, scale=None, nodes=None, heads=None):
    """Attention of a linear draft verified in place, ONE layer.

    The draft's K/V sit at positions ctx .. ctx + T - 1 after the prefix, and
    draft token i (local id, position ctx + i) attends to positions 0 .. ctx + i:
    ordinary causal attention over prefix + draft, as one target pass over the
    appended span computes it.  Shapes as in tree_attention (no tree arrays);
    ``nodes`` / ``heads`` restrict the computation, other entries are NaN.
    """
    q = _f64(q)
    kc, vc = _f64(k_cache), _f64(v_cache)
    total, n_q, d = q.shape
    n_kv = kc.shape[1]
    if n_q % n_kv:
        raise ValueError("n_q must be a multiple of n_kv")
    g = n_q // n_kv
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    node_off = np.asarray(node_off)
    want_nodes = set(range(total)) if nodes is None else set(int(x) for x in nodes)
    want_heads = list(range(n_q)) if heads is None else [int(h) for h in heads]
    out = np.full((total, n_q, d), np.nan)
    for s in range(len(node_off) - 1):
        o, T = int(node_off[s]), int(node_off[s + 1] - node_off[s])
        ctx = int(ctx_len[s])
        for hk in range(n_kv):
            hs = [h for h in want_heads if h // g == hk]
            if not hs:
                continue
            keys = _context_kv(kc, block_table[s], ctx + T, hk)
            vals = _context_kv(vc, block_table[s], ctx + T, hk)
            for i in range(T):
                if o + i not in want_nodes:
                    continue
                for h in hs:
                    sc = scale * (keys[:ctx + i + 1] @ q[o + i, h])
                    p = np.exp(sc - sc.max())
                    p /= p.sum()
                    out[o + i, h] = p @ vals[:ctx + i + 1]
    return out


def accept_chain(argmax, draft_tok, node_off, max_T=None):
    """Eq. (piecewise) on a linear draft: d_1 .. d_j are accepted for the
    largest j with decode(p_k) = d_k for every k <= j, where p_k comes from the
    logits at d_{k-1} (the root for k = 1).  Returns (accept_len = j,
    path = 0 .. j padded with -1 to max_T, bonus = argmax at d_j)."""
    argmax = np.asarray(argmax)
    draft_tok = np.asarray(draft_tok)
    node_off = np.asarray(node_off)
    B = len(node_off) - 1
    Ts = np.diff(node_off)
    if max_T is None:
        max_T = int(Ts.max())
    accept_len = np.zeros(B, dtype=np.int32)
    path = np.full((B, max_T), -1, dtype=np.int32)
    bonus = np.zeros(B, dtype=np.int32)
    for s in range(B):
        o, T = int(node_off[s]), int(Ts[s])
        j = 0
        while j + 1 < T and int(draft_tok[o + j + 1]) == int(argmax[o + j]):
            j += 1
        accept_len[s] = j
        path[s, :j + 1] = np.arange(j + 1)
        bonus[s] = int(argmax[o + j])
    return accept_len, path, bonus


# ----------------------------------------------------------------------------
# Reuse <-> Generate controller (Sec. III-A): the next draft tree from the match
# points, and the commit of a verification step's result
# ----------------------------------------------------------------------------

def build_reuse_tree(orig_tokens, orig_off, match_pos, n_matches, last_tok, n, chain_len, n_branches,
                     gen_tok=None):
    """Draft tree of the next step, every sequence.

    Sec. III-A: match points of the generated suffix in the remaining code are
    new draft starts, and the code after each of them is a draft.  Node 0 is
    the root, the last committed token.  Branch b (b < n_branches) holds the
    chain_len tokens of c after the b-th match point p_b,
    c[p_b + n + j] for j < chain_len, as a chain below the root; a branch with
    no match point, and positions past the end of c, carry token -1 (no argmax
    equals it, so such nodes are never accepted).  Then the generated branch:
    gen_tok[s] (a draft model's proposal for edited content, G tokens, G = 0
    allowed), also a chain below the root and marked in gen_mask.
    Every sequence has T = 1 + n_branches * chain_len + G nodes.

    Returns (draft_tok int32 [B*T], parent int32 [B*T] local ids,
    node_off int32 [B+1], cpos int32 [B*T] = the node's position in c
    (the root: p_0 + n - 1, its match; -1 for generated or empty nodes),
    gen_mask uint8 [B*T]).
    """
    orig_tokens = np.asarray(orig_tokens)
    orig_off = np.asarray(orig_off)
    match_pos = np.asarray(match_pos)
    B = len(orig_off) - 1
    G = 0 if gen_tok is None else np.asarray(gen_tok).shape[1]
    T = 1 + n_branches * chain_len + G
    draft = np.full(B * T, -1, np.int32)
    parent = np.zeros(B * T, np.int32)
    cpos = np.full(B * T, -1, np.int32)
    gmask = np.zeros(B * T, np.uint8)
    for s in range(B):
        o = s * T
        c = orig_tokens[orig_off[s]:orig_off[s + 1]]
        draft[o] = last_tok[s]
        parent[o] = -1
        if n_matches[s] > 0:
            cpos[o] = match_pos[s, 0] + n - 1
        for b in range(n_branches):
            has = b < min(int(n_matches[s]), match_pos.shape[1])
            for j in range(chain_len):
                i = 1 + b * chain_len + j
                parent[o + i] = 0 if j == 0 else i - 1
                if has:
                    q = int(match_pos[s, b]) + n + j
                    if q < len(c):
                        draft[o + i] = c[q]
                        cpos[o + i] = q
        for j in range(G):
            i = 1 + n_branches * chain_len + j
            parent[o + i] = 0 if j == 0 else i - 1
            draft[o + i] = gen_tok[s][j]
            gmask[o + i] = 1
    node_off = (np.arange(B + 1) * T).astype(np.int32)
    return draft, parent, node_off, cpos, gmask


def advance(out_tok, out_len, draft_tok, cpos, node_off, path, accept_len, bonus, cursor, n):
    """Commit one verification step (Sec. III-A).

    The accepted draft tokens -- path nodes 1 .. accept_len (the root was
    committed before) -- and the bonus token extend the generated sequence.
    The tail becomes its last n tokens and the root of the next tree is the
    bonus.  The cursor marks the start of the code not yet verified: when the
    last accepted node came from c (cpos q >= 0), the code up to q is consumed
    and the rest, from q + 1, stays the candidate draft; otherwise it stays.

    Returns (out_tok', out_len', tail int32 [B, n], cursor', last_tok)."""
    out = np.array(out_tok, copy=True)
    out_len = np.asarray(out_len).astype(np.int32).copy()
    cursor = np.asarray(cursor).astype(np.int32).copy()
    B = len(out_len)
    tail = np.zeros((B, n), np.int32)
    last = np.zeros(B, np.int32)
    for s in range(B):
        o = int(node_off[s])
        a = int(accept_len[s])
        toks = [int(draft_tok[o + int(path[s, k])]) for k in range(1, a + 1)] + [int(bonus[s])]
        L = int(out_len[s])
        if L + len(toks) > out.shape[1]:
            raise ValueError("committed-token buffer full")
        out[s, L:L + len(toks)] = toks
        out_len[s] = L + len(toks)
        tail[s] = out[s, out_len[s] - n:out_len[s]]
        q = int(cpos[o + int(path[s, a])])
        if q >= 0:
            cursor[s] = q + 1
        last[s] = int(bonus[s])
    return out, out_len, tail, cursor, last


# ----------------------------------------------------------------------------
# Entropy-aware dynamic verification -- Eq. (entropy) and the top_tau rule
# ----------------------------------------------------------------------------

def entropy_top_tau(logits, k, renormalize=False):
    """top_tau for one position from its full-vocabulary logits.

    Eq. (entropy): H_norm = -sum_{i<=k} p_i log p_i / log k over the k largest
    probabilities of the target distribution; top_tau = ceil(k H_norm), or 1
    when that is below 1.  Reading: p_i are the softmax probabilities over the
    whole vocabulary, not renormalised over the top k (``renormalize`` gives the
    other reading); top_tau counts top-k candidates, so it is at most k (H_norm
    <= 1 for k >= 3 in exact arithmetic; the clamp only absorbs rounding of
    H_norm = 1).  Returns (top_tau, H_norm, ranked token ids of the top k).
    """
    x = _f64(logits)
    p = np.exp(x - x.max())
    p /= p.sum()
    order = np.lexsort((np.arange(len(p)), -p))[:k]      # descending p, ties to lowest id
    pk = p[order]
    if renormalize:
        pk = pk / pk.sum()
    nz = pk[pk > 0]
    h = float(-(nz * np.log(nz)).sum() / math.log(k))
    tau = min(k, max(1, math.ceil(k * h)))
    return tau, h, order


VERIFY_MODES = ("greedy", "direct", "topk", "entropy")


def node_ranking(logits, K):
    """The K most probable tokens of one target distribution, most probable
    first; among equal probabilities (equal logits) the lower token id ranks
    first (the tie rule of decode(), reading A6)."""
    x = _f64(logits)
    return np.lexsort((np.arange(len(x)), -x))[:K]


def verify_accept(logits, draft_tok, parent, node_off, mode, k=1, gen_mask=None, max_T=None,
                  tau_override=None):
    """Longest accepted draft path under one of the verification rules the
    paper compares (Sec. V-C, RQ3), applied along every root-to-node path of
    the tree as in accept_path.

    The edge a -> b (b drafted after a) is judged on the target distribution at
    a (the logits of node a).  Edit content -- the nodes with gen_mask[b] = 1,
    every node when gen_mask is None -- is judged by ``mode``; reused code stays
    greedy (Sec. IV-E: only the edit content of EfficientEdit uses the
    entropy-aware rule, the Reuse phase verifies greedily):
      greedy   draft_tok[b] is the target's most probable token (rank 0);
      direct   accepted without verification;
      topk     draft_tok[b] ranks within the target's k most probable tokens;
      entropy  draft_tok[b] ranks within the first top_tau of them, top_tau
               from Eq. (entropy) at a (entropy_top_tau, Sec. III-B).
    Ranks order tokens by probability, lower id first among equal ones.  The
    accepted path is the deepest accepted node's root path (lowest node id
    among equally deep ones, reading A9); bonus = the target's most probable
    token at that node (Sec. II-B).

    ``tau_override`` (int array [sum T]) replaces the computed top_tau of the
    entropy rule node by node -- for checking a kernel's acceptance given its
    own top_tau where k * H_norm sits at an integer.

    Returns (accept_len int32 [B], path int32 [B, max_T], bonus int32 [B],
    tau int32 [sum T]) where tau[a] is the number of leading ranks an
    edit-content child of a may hold (greedy 1, topk k, entropy top_tau,
    direct 0 = any).
    """
    if mode not in VERIFY_MODES:
        raise ValueError(mode)
    x = _f64(logits)
    draft_tok = np.asarray(draft_tok)
    parent = np.asarray(parent)
    node_off = np.asarray(node_off)
    total = len(draft_tok)
    gen = np.ones(total, dtype=bool) if gen_mask is None else np.asarray(gen_mask).astype(bool)
    B = len(node_off) - 1
    Ts = np.diff(node_off)
    if max_T is None:
        max_T = int(Ts.max())
    kk = max(1, int(k))
    ranked = [node_ranking(x[a], max(kk, 1)) for a in range(total)]
    tau = np.zeros(total, dtype=np.int32)
    for a in range(total):
        if mode == "greedy":
            tau[a] = 1
        elif mode == "topk":
            tau[a] = kk
        elif mode == "entropy":
            tau[a] = entropy_top_tau(x[a], kk)[0] if tau_override is None else int(tau_override[a])
    accept_len = np.zeros(B, dtype=np.int32)
    path = np.full((B, max_T), -1, dtype=np.int32)
    bonus = np.zeros(B, dtype=np.int32)
    for s in range(B):
        o, T = int(node_off[s]), int(Ts[s])
        accepted = [False] * T
        depth = [0] * T
        accepted[0] = True
        for i in range(1, T):
            p = int(parent[o + i])
            depth[i] = depth[p] + 1
            a, tok = o + p, int(draft_tok[o + i])
            if not gen[o + i]:
                ok = tok == int(ranked[a][0])                      # reused code: greedy
            elif mode == "direct":
                ok = True
            else:
                ok = tok in [int(t) for t in ranked[a][:int(tau[a])]]
            accepted[i] = accepted[p] and ok
        best = 0
        for i in range(1, T):
            if accepted[i] and depth[i] > depth[best]:
                best = i
        chain = []
        u = best
        while u != -1:
            chain.append(u)
            u = int(parent[o + u]) if u != 0 else -1
        chain.reverse()
        accept_len[s] = depth[best]
        path[s, :len(chain)] = chain
        bonus[s] = int(ranked[o + best][0])
    return accept_len, path, bonus, tau


# ----------------------------------------------------------------------------
# one whole step
# ----------------------------------------------------------------------------

def verify_step(w, layers=None, vocab_rows=None):
    """The whole verification step on a workload (workloads.Workload): match,
    tree structure, attention for the requested layers, LM head + argmax,
    acceptance and compaction.  ``vocab_rows`` (a slice) restricts the LM head
    to part of the vocabulary, for bounded CPU timing only."""
    res = {}
    res["match_pos"], res["n_matches"] = match_reuse(w.orig_tokens, w.orig_off, w.tail, w.cursor,
                                                     w.max_matches)
    depth, anc = tree_prepare(w.parent, w.node_off)
    res["depth"], res["anc"] = depth, anc
    layers = range(w.layers) if layers is None else layers
    res["attn"] = {l: tree_attention(w.q[l], w.k_tree[l], w.v_tree[l], w.k_cache[l], w.v_cache[l],
                                     w.block_table, w.ctx_len, w.node_off, anc) for l in layers}
    if vocab_rows is None:
        am, _, _ = lm_head_argmax(w.hidden_states, w.lm_w)
    else:
        logits, _ = lm_head_logits(w.hidden_states, w.lm_w, rows=vocab_rows)
        am = (np.argmax(logits, axis=1) + (vocab_rows.start or 0)).astype(np.int32)
    res["argmax"] = am
    acc, path, bonus = accept_path(am, w.draft_tok, w.parent, w.node_off, w.max_T)
    res["accept_len"], res["path"], res["bonus"] = acc, path, bonus
    lay = list(layers)
    res["k_cache"], res["v_cache"], res["dst_slot"], res["ctx_out"] = kv_compact(
        _raw16(w.k_tree[lay]), _raw16(w.v_tree[lay]), _raw16(w.k_cache[lay]), _raw16(w.v_cache[lay]),
        w.block_table, w.ctx_len, w.node_off, path, acc)
    return res
