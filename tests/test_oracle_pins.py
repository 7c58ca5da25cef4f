"""Pins of the fp64 oracle to facts outside itself (CPU only).

Each test checks an oracle function against something it does not contain:
hand-worked golden cases (tests/golden/, each citing its equation), a brute
force written a different way, a library routine on a special case, a closed
form, or an answer the input generator planted.  A plausible slip in the
oracle -- a dropped term, a wrong sign, an off-by-one, a transposed operand, a
wrong GQA head map -- fails at least one of them.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle as O
import workloads as W

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _gold(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _bf16_np(t):
    return t.detach().cpu().double().numpy()


# ----------------------------------------------------------------------------
# match
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("case", _gold("match_cases.json")["cases"], ids=lambda c: c["name"])
def test_match_golden(case):
    c = np.asarray(case["c"], dtype=np.int32)
    tail = np.asarray([case["tail"]], dtype=np.int32)
    pos, cnt = O.match_reuse(c, np.asarray([0, len(c)]), tail, np.asarray([case["cursor"]]), 4)
    k = case["n_matches"]
    assert cnt[0] == k
    assert list(pos[0, :min(k, 4)]) == case["match_pos"][:4]
    assert np.all(pos[0, min(k, 4):] == -1)


def _bytes_find_all(c, tail, cursor):
    """Brute force by a different route: byte-string search over 4-byte tokens."""
    hay = np.asarray(c, dtype=">i4").tobytes()
    needle = np.asarray(tail, dtype=">i4").tobytes()
    out, start = [], 0
    while True:
        i = hay.find(needle, start)
        if i < 0:
            break
        if i % 4 == 0:
            p = i // 4
            if p >= cursor and p + len(tail) < len(c):
                out.append(p)
        start = i + 1
    return out


@pytest.mark.parametrize("n", [2, 4, 8])
def test_match_bruteforce_sweep(n):
    w = W.build("sweep", B=6, layers=1, n=n, seed=77 + n)
    pos, cnt = O.match_reuse(w.orig_tokens, w.orig_off, w.tail, w.cursor, 5)
    for s in range(w.B):
        ref = _bytes_find_all(w.seq_tokens(s), w.tail[s], int(w.cursor[s]))
        assert cnt[s] == len(ref)
        assert list(pos[s, :min(5, len(ref))]) == ref[:5]
        if w.planted_match[s] >= 0:
            assert w.planted_match[s] in ref or len(ref) > 5


def test_match_closed_form_constant_code():
    L, n = 50, 3
    c = np.full(L, 9, dtype=np.int32)
    for cur in [0, 5, 46, 47, 60]:
        pos, cnt = O.match_reuse(c, np.asarray([0, L]), np.full((1, n), 9, np.int32), np.asarray([cur]), 64)
        # every p with cur <= p <= L - n - 1 matches
        want = list(range(cur, L - n))
        assert cnt[0] == len(want)
        assert list(pos[0, :len(want)]) == want


def test_match_planted_tiny():
    w = W.build("tiny")
    pos, cnt = O.match_reuse(w.orig_tokens, w.orig_off, w.tail, w.cursor, w.max_matches)
    assert pos[0, 0] == w.planted_match[0] == 296
    # the reuse chain the generator built starts at the last matched token
    c = w.seq_tokens(0)
    p, n = int(pos[0, 0]), w.n
    assert list(w.draft_tok[:12]) == list(c[p + n - 1:p + n + 11])


def test_match_rejects_bad_args():
    with pytest.raises(ValueError):
        O.match_reuse(np.arange(5, dtype=np.int32), np.asarray([0, 5]), np.zeros((1, 2), np.int32),
                      np.asarray([-1]), 2)


# ----------------------------------------------------------------------------
# tree structure
# ----------------------------------------------------------------------------

def _walk_up(parent, o, i):
    path = []
    u = i
    while u != -1:
        path.append(u)
        u = int(parent[o + u])
    return path[::-1]


def test_tree_prepare_closed_forms():
    chain = np.asarray([-1] + list(range(127)), dtype=np.int32)
    star = np.asarray([-1] + [0] * 9, dtype=np.int32)
    parent = np.concatenate([chain, star])
    off = np.asarray([0, 128, 138])
    depth, anc = O.tree_prepare(parent, off)
    for i in range(128):
        assert depth[i] == i
        assert O.anc_to_sets(anc[i]) == set(range(i + 1))
    for i in range(10):
        assert depth[128 + i] == (0 if i == 0 else 1)
        assert O.anc_to_sets(anc[128 + i]) == ({0} if i == 0 else {0, i})
    # bit layout: node 127 of the chain sets every bit of both words
    assert int(anc[127, 0]) == 2 ** 64 - 1 and int(anc[127, 1]) == 2 ** 64 - 1


def test_tree_prepare_walk_up():
    w = W.build("batched", layers=1, vocab=512, hidden=64, seed=5)
    depth, anc = O.tree_prepare(w.parent, w.node_off)
    for s in range(w.B):
        o, T = int(w.node_off[s]), int(w.node_off[s + 1] - w.node_off[s])
        for i in range(T):
            p = _walk_up(w.parent, o, i)
            assert depth[o + i] == len(p) - 1
            assert O.anc_to_sets(anc[o + i]) == set(p)


@pytest.mark.parametrize("parent", [[0, 0], [-1, 1], [-1, 0, 3, 1], [-1, -1]])
def test_tree_prepare_rejects(parent):
    with pytest.raises(ValueError):
        O.tree_prepare(np.asarray(parent, np.int32), np.asarray([0, len(parent)]))


# ----------------------------------------------------------------------------
# attention
# ----------------------------------------------------------------------------

def _linear_kv(w, layer, s, hk, path_nodes, cache):
    """Keys (or values) of the linear sequence context + path, gathered one position
    at a time through the block table."""
    kc, kt = (w.k_cache, w.k_tree) if cache == "k" else (w.v_cache, w.v_tree)
    rows = []
    for pos in range(int(w.ctx_len[s])):
        page = int(w.block_table[s, pos // W.PAGE])
        rows.append(kc[layer, page, hk, pos % W.PAGE])
    o = int(w.node_off[s])
    for j in path_nodes:
        rows.append(kt[layer, o + j, hk])
    return torch.stack(rows).double()


def _sdpa_last(qv, keys, vals):
    """torch SDPA (fp64, math backend) for one query vector at the end of a sequence."""
    return F.scaled_dot_product_attention(qv[None, None, None, :], keys[None, None], vals[None, None])[0, 0, 0]


@pytest.mark.parametrize("q_std", [1.0, 40.0])
def test_attention_each_node_is_causal_attention_over_its_path(q_std):
    tree = W.TreeSpec(6, [(0, 3), (3, 2)], [0, 1, 2])
    w = W.build("tiny", ctx=37, trees=[tree, W.TreeSpec(3, [(1, 2)], [0])], q_std=q_std)
    depth, anc = O.tree_prepare(w.parent, w.node_off)
    out = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0],
                           w.block_table, w.ctx_len, w.node_off, anc)
    g = w.n_q // w.n_kv
    for s in range(w.B):
        o, T = int(w.node_off[s]), int(w.node_off[s + 1] - w.node_off[s])
        for i in range(T):
            path = _walk_up(w.parent, o, i)
            for h in range(w.n_q):
                keys = _linear_kv(w, 0, s, h // g, path, "k")
                vals = _linear_kv(w, 0, s, h // g, path, "v")
                ref = _sdpa_last(w.q[0, o + i, h].double(), keys, vals).numpy()
                np.testing.assert_allclose(out[o + i, h], ref, rtol=0, atol=1e-12)


def test_attention_chain_equals_masked_sdpa():
    """A chain-only tree is the paper's linear draft: causal attention over ctx + T."""
    w = W.build("tiny", ctx=45, trees=[W.TreeSpec(9, [], [0, 1])])
    depth, anc = O.tree_prepare(w.parent, w.node_off)
    out = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0],
                           w.block_table, w.ctx_len, w.node_off, anc)
    T, ctx, g = 9, 45, w.n_q // w.n_kv
    keys = torch.stack([_linear_kv(w, 0, 0, hk, range(T), "k") for hk in range(w.n_kv)])
    vals = torch.stack([_linear_kv(w, 0, 0, hk, range(T), "v") for hk in range(w.n_kv)])
    keys = keys.repeat_interleave(g, dim=0)        # [n_q, ctx+T, d]
    vals = vals.repeat_interleave(g, dim=0)
    qq = w.q[0, :T].double().permute(1, 0, 2)      # [n_q, T, d]
    mask = torch.arange(ctx + T)[None, :] <= (ctx + torch.arange(T))[:, None]
    ref = F.scaled_dot_product_attention(qq[None], keys[None], vals[None], attn_mask=mask)[0]
    np.testing.assert_allclose(out[:T], ref.permute(1, 0, 2).numpy(), rtol=0, atol=1e-12)


def test_attention_single_key_returns_value():
    """T = 1 and ctx = 0: softmax over one key is 1, the output is that value row."""
    w = W.build("tiny", ctx=0, trees=[W.TreeSpec(1, [], [0])])
    depth, anc = O.tree_prepare(w.parent, w.node_off)
    out = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0],
                           w.block_table, w.ctx_len, w.node_off, anc)
    g = w.n_q // w.n_kv
    for h in range(w.n_q):
        assert np.array_equal(out[0, h], _bf16_np(w.v_tree[0, 0, h // g]))


def test_attention_equal_keys_average_values():
    """All keys equal: the softmax is uniform and the output is the plain mean of the values."""
    w = W.build("tiny", ctx=21, trees=[W.TreeSpec(4, [(1, 2)], [0])])
    w.k_cache[:] = 0.25
    w.k_tree[:] = 0.25
    depth, anc = O.tree_prepare(w.parent, w.node_off)
    out = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0],
                           w.block_table, w.ctx_len, w.node_off, anc)
    g = w.n_q // w.n_kv
    node = 5                              # second node of the branch hanging off node 1
    path = _walk_up(w.parent, 0, node)
    for h in range(w.n_q):
        vals = _linear_kv(w, 0, 0, h // g, path, "v").numpy()
        np.testing.assert_allclose(out[node, h], vals.mean(axis=0), rtol=0, atol=1e-14)


def test_attention_page_order_invariance():
    w = W.build("tiny", ctx=70)
    depth, anc = O.tree_prepare(w.parent, w.node_off)
    args = (w.block_table, w.ctx_len, w.node_off, anc)
    ref = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0], *args)
    rng = np.random.default_rng(3)
    perm = rng.permutation(w.num_pages)                 # new page p' = perm[p]
    kc = torch.empty_like(w.k_cache[0])
    vc = torch.empty_like(w.v_cache[0])
    kc[torch.as_tensor(perm)] = w.k_cache[0]
    vc[torch.as_tensor(perm)] = w.v_cache[0]
    bt = np.where(w.block_table >= 0, perm[np.maximum(w.block_table, 0)], -1).astype(np.int32)
    got = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], kc, vc, bt, w.ctx_len, w.node_off, anc)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-13)


def test_attention_gqa_head_map():
    """Query head h reads KV head h // g: perturbing KV head 1 moves heads g..2g-1 only."""
    w = W.build("tiny", ctx=33)
    depth, anc = O.tree_prepare(w.parent, w.node_off)
    args = (w.block_table, w.ctx_len, w.node_off, anc)
    ref = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0], *args)
    vc = w.v_cache[0].clone()
    vc[:, 1] += 1.0
    got = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], vc, *args)
    g = w.n_q // w.n_kv
    moved = np.abs(got - ref).max(axis=(0, 2)) > 1e-6
    assert list(np.nonzero(moved)[0]) == list(range(g, 2 * g))


# ----------------------------------------------------------------------------
# LM head and argmax
# ----------------------------------------------------------------------------

def test_lm_head_pure_python_dot():
    w = W.build("tiny", vocab=37, hidden=24, trees=[W.TreeSpec(3, [], [0])])
    logits, err = O.lm_head_logits(w.hidden_states, w.lm_w)
    x = w.hidden_states.double().tolist()
    wt = w.lm_w.double().tolist()
    for i in range(len(x)):
        for v in range(37):
            ref = math.fsum(a * b for a, b in zip(x[i], wt[v]))
            assert abs(logits[i, v] - ref) <= 1e-12 * (1 + abs(ref))
            assert err[i, v] >= 0


@pytest.mark.parametrize("name,ov", [("tiny", {}), ("7b", dict(layers=1, vocab=8192, hidden=768)),
                                     ("batched", dict(layers=1, vocab=6000, hidden=320))])
def test_lm_head_planted_argmax(name, ov):
    w = W.build(name, **ov)
    am, cands, _ = O.lm_head_argmax(w.hidden_states, w.lm_w)
    planted = w.planted_argmax >= 0
    assert planted.sum() > 0
    np.testing.assert_array_equal(am[planted], w.planted_argmax[planted])
    for i in np.nonzero(planted)[0]:
        assert list(cands[i]) == [w.planted_argmax[i]]


def test_lm_head_duplicate_rows_lowest_id():
    w = W.build("tiny", dup_rows=3)
    am, cands, logits = O.lm_head_argmax(w.hidden_states, w.lm_w)
    planted = w.planted_argmax >= 0
    np.testing.assert_array_equal(am[planted], w.planted_argmax[planted])
    tied = [i for i in np.nonzero(planted)[0] if len(cands[i]) > 1]
    assert tied, "duplicated rows must create exact ties"
    for i in tied:
        top = np.nonzero(logits[i] == logits[i].max())[0]
        assert len(top) == 2 and am[i] == top.min()


def test_lm_head_fp32_accumulation_stays_within_the_bound():
    """Reading A7's bound holds for fp32 accumulation in any order: products of
    two bf16 values are exact in fp32, and the sum of H rounded additions is off
    by at most 2 H 2^-24 sum_k |x_k w_k| whatever the order (sequential, reversed,
    16-wide blocks with fp32 partial sums as a tensor core forms them, BLAS)."""
    H, V, n = 1024, 96, 3
    g = torch.Generator().manual_seed(7)
    x = torch.randn(n, H, generator=g).to(torch.bfloat16)
    wm = (0.02 * torch.randn(V, H, generator=g)).to(torch.bfloat16)
    logits, err = O.lm_head_logits(x, wm)
    xf = x.float().numpy()
    wf = wm.float().numpy()
    prods = xf[:, None, :] * wf[None, :, :]                   # exact in fp32
    orders = {}
    acc = np.zeros((n, V), np.float32)
    for k in range(H):
        acc = (acc + prods[:, :, k]).astype(np.float32)
    orders["sequential"] = acc
    acc = np.zeros((n, V), np.float32)
    for k in reversed(range(H)):
        acc = (acc + prods[:, :, k]).astype(np.float32)
    orders["reversed"] = acc
    acc = np.zeros((n, V), np.float32)
    for k0 in range(0, H, 16):
        part = np.zeros((n, V), np.float32)
        for k in range(k0, k0 + 16):
            part = (part + prods[:, :, k]).astype(np.float32)
        acc = (acc + part).astype(np.float32)
    orders["blocked16"] = acc
    orders["blas"] = (xf @ wf.T).astype(np.float32)
    for name, y in orders.items():
        dev = np.abs(y.astype(np.float64) - logits)
        assert np.all(dev <= err), f"{name}: fp32 logits leave the bound by {(dev - err).max():.3e}"
    assert err.max() < 1e-3 * np.abs(logits).max() + 1e-3    # and the bound is far from vacuous


def test_lm_head_candidates_hold_every_argmax_within_the_bound():
    """Any logits within err of the fp64 ones have their argmax among the
    candidates -- including adversarial ones that raise a runner-up by err and
    lower the maximum by err."""
    rng = np.random.default_rng(3)
    w = W.build("tiny", vocab=300, hidden=64, trees=[W.TreeSpec(6, [], [0])])
    am, cands, logits = O.lm_head_argmax(w.hidden_states, w.lm_w)
    _, err = O.lm_head_logits(w.hidden_states, w.lm_w)
    for i in range(logits.shape[0]):
        top = int(np.argmax(logits[i]))
        for _ in range(50):
            y = logits[i] + err[i] * rng.uniform(-1, 1, size=logits.shape[1])
            assert int(np.argmax(y)) in set(cands[i].tolist())
        for v in range(logits.shape[1]):
            y = logits[i].copy()
            y[top] -= err[i, top]
            y[v] += err[i, v]
            if int(np.argmax(y)) == v:
                assert v in set(cands[i].tolist())


def test_lm_head_candidates_at_a_gap_between_one_and_two_bounds():
    """Hand-built near ties (H = 64, x = all ones, rows of ones differing in
    element 0): the bound is err = 2 H 2^-24 sum_k |w_k| ~ 4.8e-4 per logit.
    Row b trails row a by 2^-10 - 2^-12 = 7.3e-4: more than one bound, less
    than two, so fp32 results may swap them and b is a candidate.  Row c
    trails by 2^-10 + 2^-9 = 2.9e-3, more than both bounds: never the argmax."""
    H = 64
    x = torch.ones(1, H, dtype=torch.bfloat16)
    w = torch.ones(4, H, dtype=torch.float32)
    w[0, 0], w[1, 0], w[2, 0], w[3, 0] = -1.0, 2.0 ** -10, 2.0 ** -12, -(2.0 ** -9)   # rows: z, a, b, c
    w = w.to(torch.bfloat16)
    am, cands, logits = O.lm_head_argmax(x, w)
    _, err = O.lm_head_logits(x, w)
    gap_b, gap_c = logits[0, 1] - logits[0, 2], logits[0, 1] - logits[0, 3]
    assert err[0, 1] < gap_b < err[0, 1] + err[0, 2] and gap_c > err[0, 1] + err[0, 3]
    assert am[0] == 1 and list(cands[0]) == [1, 2]


def test_lm_head_identity_closed_form():
    """W rows = unit vectors e_v (v < H): logits are the hidden coordinates."""
    H = 64
    x = torch.randn(5, H, generator=torch.Generator().manual_seed(0)).to(torch.bfloat16)
    wmat = torch.eye(H, dtype=torch.bfloat16)
    am, cands, logits = O.lm_head_argmax(x, wmat)
    np.testing.assert_array_equal(logits, x.double().numpy())
    np.testing.assert_array_equal(am, np.argmax(x.double().numpy(), axis=1))


# ----------------------------------------------------------------------------
# acceptance
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("case", _gold("accept_cases.json")["cases"], ids=lambda c: c["name"])
def test_accept_golden(case):
    parent = np.asarray(case["parent"], np.int32)
    off = np.asarray([0, len(parent)])
    acc, path, bonus = O.accept_path(np.asarray(case["argmax"]), np.asarray(case["draft_tok"]), parent, off)
    assert acc[0] == case["accept_len"]
    assert list(path[0, :acc[0] + 1]) == case["path"]
    assert np.all(path[0, acc[0] + 1:] == -1)
    assert bonus[0] == case["bonus"]


def _replay_chain(argmax, draft):
    """Eq. (piecewise) read literally: largest j with decode(p_i) == d_i for all i <= j."""
    j = 0
    while j + 1 < len(draft) and argmax[j] == draft[j + 1]:
        j += 1
    return j


def _brute_longest(argmax, draft, parent):
    """Every root-to-node path checked by replay; deepest accepted node, lowest id."""
    best, best_len = 0, 0
    for u in range(len(parent)):
        path = _walk_up(parent, 0, u)
        ok = all(draft[b] == argmax[a] for a, b in zip(path[:-1], path[1:]))
        if ok and len(path) - 1 > best_len:
            best, best_len = u, len(path) - 1
    return best, best_len


def test_accept_chain_replay_random():
    rng = np.random.default_rng(11)
    for _ in range(300):
        T = int(rng.integers(1, 40))
        draft = rng.integers(0, 3, size=T)
        am = rng.integers(0, 3, size=T)
        parent = np.asarray([-1] + list(range(T - 1)), np.int32)
        acc, path, bonus = O.accept_path(am, draft, parent, np.asarray([0, T]))
        j = _replay_chain(am, draft)
        assert acc[0] == j and list(path[0, :j + 1]) == list(range(j + 1)) and bonus[0] == am[j]


def test_accept_tree_bruteforce_random():
    rng = np.random.default_rng(12)
    for _ in range(300):
        T = int(rng.integers(1, 30))
        parent = np.asarray([-1] + [int(rng.integers(0, i)) for i in range(1, T)], np.int32)
        draft = rng.integers(0, 3, size=T)          # small alphabet: equal siblings happen
        am = rng.integers(0, 3, size=T)
        acc, path, bonus = O.accept_path(am, draft, parent, np.asarray([0, T]))
        u, d = _brute_longest(am, draft, parent)
        assert acc[0] == d
        assert list(path[0, :d + 1]) == _walk_up(parent, 0, u)
        assert bonus[0] == am[u]


@pytest.mark.parametrize("name", ["tiny", "7b", "batched", "33b"])
def test_accept_planted(name):
    w = W.build(name, layers=1, vocab=4096, hidden=256) if name != "tiny" else W.build(name)
    am = np.where(w.planted_argmax >= 0, w.planted_argmax, -7)
    acc, path, bonus = O.accept_path(am, w.draft_tok, w.parent, w.node_off)
    np.testing.assert_array_equal(acc, w.planted_accept)
    for s in range(w.B):
        assert list(path[s, :acc[s] + 1]) == w.planted_path[s]


# ----------------------------------------------------------------------------
# compaction
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("case", _gold("compact_cases.json")["cases"], ids=lambda c: c["name"])
def test_compact_golden(case):
    L, n_kv, d, T = 2, 2, 4, 8
    npg = max(case["block_table"]) + 1
    kt = np.arange(L * T * n_kv * d, dtype=np.float64).reshape(L, T, n_kv, d)
    vt = -kt
    kc = np.zeros((L, npg, n_kv, 16, d))
    vc = np.zeros_like(kc)
    path = np.full((1, T), -1, np.int32)
    path[0, :len(case["path"])] = case["path"]
    kc2, vc2, dst, ctx_out = O.kv_compact(kt, vt, kc, vc, np.asarray([case["block_table"]]),
                                          np.asarray([case["ctx"]]), np.asarray([0, T]), path,
                                          np.asarray([case["accept_len"]]))
    assert list(dst[0, :len(case["dst_slot"])]) == case["dst_slot"]
    assert ctx_out[0] == case["ctx_out"]
    for k, slot in enumerate(case["dst_slot"]):
        np.testing.assert_array_equal(kc2[:, slot // 16, :, slot % 16], kt[:, case["path"][k]])
        np.testing.assert_array_equal(vc2[:, slot // 16, :, slot % 16], vt[:, case["path"][k]])


def test_compact_sequential_append_and_canary():
    w = W.build("sweep", B=5, layers=2, seed=9)
    kt = w.k_tree.view(torch.int16).numpy()
    vt = w.v_tree.view(torch.int16).numpy()
    kc = w.k_cache.view(torch.int16).numpy()
    vc = w.v_cache.view(torch.int16).numpy()
    T = w.max_T
    path = np.full((w.B, T), -1, np.int32)
    for s in range(w.B):
        path[s, :len(w.planted_path[s])] = w.planted_path[s]
    kc2, vc2, dst, ctx_out = O.kv_compact(kt, vt, kc, vc, w.block_table, w.ctx_len, w.node_off, path,
                                          w.planted_accept)
    # independent: a dict of slots filled by appending, position by position
    slots = {}
    for s in range(w.B):
        pos = int(w.ctx_len[s])
        for node in w.planted_path[s]:
            page = int(w.block_table[s, pos // 16])
            slots[(page, pos % 16)] = int(w.node_off[s]) + node
            pos += 1
        assert ctx_out[s] == pos
    for (page, off), src in slots.items():
        assert np.array_equal(kc2[:, page, :, off], kt[:, src])
        assert np.array_equal(vc2[:, page, :, off], vt[:, src])
    # canary: every other slot keeps its bytes
    keep = np.ones((w.num_pages, 16), bool)
    for (page, off) in slots:
        keep[page, off] = False
    def by_slot(a):
        return a.transpose(0, 1, 3, 2, 4)[:, keep]      # [L, pages, PAGE, n_kv, d] -> kept slots
    assert np.array_equal(by_slot(kc2), by_slot(kc)) and np.array_equal(by_slot(vc2), by_slot(vc))


# ----------------------------------------------------------------------------
# entropy-aware verification (Eq. (entropy))
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("case", _gold("entropy_cases.json")["cases"], ids=lambda c: c["name"])
def test_entropy_golden(case):
    p = np.asarray(case["probs"])
    with np.errstate(divide="ignore"):
        logits = np.where(p > 0, np.log(np.where(p > 0, p, 1.0)), -np.inf)
    tau, h, order = O.entropy_top_tau(logits, case["k"])
    assert tau == case["top_tau"]
    assert abs(h - case["h_norm"]) < 1e-5
    assert p[order[0]] == p.max()


# ----------------------------------------------------------------------------
# verification rules (Sec. V-C: Greedy / Direct / Top-k / Entropy)
# ----------------------------------------------------------------------------

def _rank(x, tok):
    """Rank of token tok in one distribution, counted: tokens with a higher logit,
    plus tokens with an equal logit and a lower id."""
    return sum(1 for v in range(len(x)) if x[v] > x[tok] or (x[v] == x[tok] and v < tok))


def _random_case(rng, T, V, levels=4):
    parent = np.asarray([-1] + [int(rng.integers(0, i)) for i in range(1, T)], np.int32)
    logits = rng.integers(0, levels, size=(T, V)).astype(np.float64)   # few levels: ties happen
    draft = rng.integers(0, V, size=T)
    gen = rng.integers(0, 2, size=T)
    return parent, logits, draft, gen


def test_verify_greedy_is_accept_path():
    rng = np.random.default_rng(21)
    for _ in range(200):
        T = int(rng.integers(1, 25))
        parent, x, draft, gen = _random_case(rng, T, 5)
        off = np.asarray([0, T])
        am = np.argmax(x, axis=1)                              # first maximum = lowest id
        ref = O.accept_path(am, draft, parent, off)
        for g in (None, gen):
            got = O.verify_accept(x, draft, parent, off, "greedy", gen_mask=g)
            for r, q in zip(ref, got[:3]):
                np.testing.assert_array_equal(r, q)


def test_verify_top1_is_greedy_and_reuse_only_is_greedy():
    rng = np.random.default_rng(22)
    for _ in range(200):
        T = int(rng.integers(1, 25))
        parent, x, draft, gen = _random_case(rng, T, 6)
        off = np.asarray([0, T])
        greedy = O.verify_accept(x, draft, parent, off, "greedy", gen_mask=gen)[:3]
        top1 = O.verify_accept(x, draft, parent, off, "topk", k=1, gen_mask=gen)[:3]
        for r, q in zip(greedy, top1):
            np.testing.assert_array_equal(r, q)
        zero = np.zeros(T, int)
        ref = O.accept_path(np.argmax(x, axis=1), draft, parent, off)     # all reused: greedy
        for mode, k in (("direct", 1), ("topk", 3), ("entropy", 3)):
            got = O.verify_accept(x, draft, parent, off, mode, k=k, gen_mask=zero)[:3]
            for r, q in zip(ref, got):
                np.testing.assert_array_equal(r, q)


def test_verify_top_vocab_is_direct():
    rng = np.random.default_rng(23)
    V = 6
    for _ in range(200):
        T = int(rng.integers(1, 25))
        parent, x, draft, gen = _random_case(rng, T, V)
        off = np.asarray([0, T])
        a = O.verify_accept(x, draft, parent, off, "topk", k=V, gen_mask=gen)[:3]
        b = O.verify_accept(x, draft, parent, off, "direct", gen_mask=gen)[:3]
        for r, q in zip(a, b):
            np.testing.assert_array_equal(r, q)


@pytest.mark.parametrize("mode,k", [("topk", 2), ("topk", 3), ("entropy", 3), ("entropy", 5),
                                    ("direct", 1), ("greedy", 1)])
def test_verify_bruteforce_random(mode, k):
    """Every root-to-node path checked edge by edge with counted ranks; the
    entropy rule's top_tau comes from its own (separately pinned) function."""
    rng = np.random.default_rng(24 + k)
    for _ in range(150):
        T = int(rng.integers(1, 20))
        V = int(rng.integers(2, 9))
        parent, x, draft, gen = _random_case(rng, T, V)
        off = np.asarray([0, T])
        acc, path, bonus, tau = O.verify_accept(x, draft, parent, off, mode, k=k, gen_mask=gen)
        def edge_ok(a, b):
            if not gen[b]:
                return _rank(x[a], draft[b]) == 0
            if mode == "direct":
                return True
            lim = {"greedy": 1, "topk": k}.get(mode)
            if lim is None:
                lim = O.entropy_top_tau(x[a], k)[0]
            return _rank(x[a], draft[b]) < lim
        best, best_len = 0, 0
        for u in range(T):
            pth = _walk_up(parent, 0, u)
            if all(edge_ok(a, b) for a, b in zip(pth[:-1], pth[1:])) and len(pth) - 1 > best_len:
                best, best_len = u, len(pth) - 1
        assert acc[0] == best_len
        assert list(path[0, :best_len + 1]) == _walk_up(parent, 0, best)
        assert bonus[0] == int(np.argmax(x[best]))


def test_verify_entropy_closed_forms():
    """H_norm = 0 (one dominant token) gives top_tau = 1, the greedy rule; k equal
    probabilities and nothing else give H_norm = 1, top_tau = k, the top-k rule."""
    V, k = 12, 4
    T = 6
    parent = np.asarray([-1, 0, 1, 2, 3, 4], np.int32)
    off = np.asarray([0, T])
    draft = np.asarray([0, 3, 2, 1, 0, 2])            # ranks 3, 2, 1, 0, 2 of the uniform top-4
    uniform = np.full((T, V), -np.inf)
    uniform[:, :k] = 0.0                               # p = 1/k on tokens 0..k-1
    onehot = np.full((T, V), -np.inf)
    onehot[:, 0] = 0.0
    acc_u, _, _, tau_u = O.verify_accept(uniform, draft, parent, off, "entropy", k=k)
    acc_t = O.verify_accept(uniform, draft, parent, off, "topk", k=k)[0]
    assert list(tau_u) == [k] * T and acc_u[0] == acc_t[0] == T - 1
    acc_o, _, _, tau_o = O.verify_accept(onehot, draft, parent, off, "entropy", k=k)
    acc_g = O.verify_accept(onehot, draft, parent, off, "greedy")[0]
    assert list(tau_o) == [1] * T and acc_o[0] == acc_g[0] == 0


# ----------------------------------------------------------------------------
# whole step on the tiny configuration
# ----------------------------------------------------------------------------

def test_verify_step_tiny_planted():
    w = W.build("tiny")
    r = O.verify_step(w)
    assert r["match_pos"][0, 0] == 296
    assert r["accept_len"][0] == w.planted_accept[0] == 7
    assert list(r["path"][0, :8]) == list(range(8))
    assert r["ctx_out"][0] == 512 + 8
    assert r["bonus"][0] == w.planted_argmax[7]
    assert not np.isnan(r["attn"][0]).any()


# ----------------------------------------------------------------------------
# in-place speculative K/V: tree K/V at positions ctx + i, compaction by moves
# ----------------------------------------------------------------------------

def _inplace_case(seed, B=4, L=2, n_kv=2, d=4):
    """Random trees (parent[i] drawn below i), a root-to-node path per tree,
    ragged contexts (not page-aligned) and a shuffled block table."""
    rng = np.random.default_rng(seed)
    Ts = [int(rng.integers(1, 40)) for _ in range(B)]
    ctx = np.asarray([int(rng.integers(0, 70)) for _ in range(B)], np.int32)
    node_off = np.concatenate([[0], np.cumsum(Ts)]).astype(np.int32)
    max_T = max(Ts)
    max_pages = (int(ctx.max()) + max_T + 15) // 16 + 1
    num_pages = B * max_pages
    bt = rng.permutation(num_pages).astype(np.int32).reshape(B, max_pages)
    path = np.full((B, max_T), -1, np.int32)
    acc = np.zeros(B, np.int32)
    for s, T in enumerate(Ts):
        parent = [-1] + [int(rng.integers(0, i)) for i in range(1, T)]
        u = int(rng.integers(0, T))
        p = [u]
        while parent[p[-1]] >= 0:
            p.append(parent[p[-1]])
        p = p[::-1]
        path[s, :len(p)] = p
        acc[s] = len(p) - 1
    total = int(node_off[-1])
    kt = rng.standard_normal((L, total, n_kv, d))
    vt = rng.standard_normal((L, total, n_kv, d))
    kc = rng.standard_normal((L, num_pages, n_kv, 16, d))
    vc = rng.standard_normal((L, num_pages, n_kv, 16, d))
    return dict(kt=kt, vt=vt, kc=kc, vc=vc, bt=bt, ctx=ctx, node_off=node_off, path=path, acc=acc,
                Ts=Ts)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_tree_kv_placement_round_trip(seed):
    c = _inplace_case(seed)
    kc2, vc2 = O.tree_kv_to_cache(c["kt"], c["vt"], c["kc"], c["vc"], c["bt"], c["ctx"], c["node_off"])
    # independent placement: a dict of slots, node by node
    slots = {}
    for s, T in enumerate(c["Ts"]):
        for i in range(T):
            pos = int(c["ctx"][s]) + i
            slots[(int(c["bt"][s, pos // 16]), pos % 16)] = int(c["node_off"][s]) + i
    for (page, off), src in slots.items():
        np.testing.assert_array_equal(kc2[:, page, :, off], c["kt"][:, src])
        np.testing.assert_array_equal(vc2[:, page, :, off], c["vt"][:, src])
    keep = np.ones(c["kc"].shape[1:2] + (16,), bool)
    for (page, off) in slots:
        keep[page, off] = False
    tk = c["kc"].transpose(0, 1, 3, 2, 4)
    assert np.array_equal(kc2.transpose(0, 1, 3, 2, 4)[:, keep], tk[:, keep])
    kt2, vt2 = O.tree_kv_from_cache(kc2, vc2, c["bt"], c["ctx"], c["node_off"])
    np.testing.assert_array_equal(kt2, c["kt"])
    np.testing.assert_array_equal(vt2, c["vt"])


@pytest.mark.parametrize("seed", [3, 4, 5, 6, 7])
def test_compact_inplace_equals_append(seed):
    """With the tree's K/V placed at ctx + i, moving the path down gives the
    cache kv_compact's append gives, on every position up to ctx + acc, and
    leaves the context untouched."""
    c = _inplace_case(seed)
    placed_k, placed_v = O.tree_kv_to_cache(c["kt"], c["vt"], c["kc"], c["vc"], c["bt"], c["ctx"],
                                            c["node_off"])
    ik, iv, idst, ictx = O.kv_compact_inplace(placed_k, placed_v, c["bt"], c["ctx"], c["node_off"],
                                              c["path"], c["acc"])
    ak, av, adst, actx = O.kv_compact(c["kt"], c["vt"], c["kc"], c["vc"], c["bt"], c["ctx"],
                                      c["node_off"], c["path"], c["acc"])
    np.testing.assert_array_equal(idst, adst)
    np.testing.assert_array_equal(ictx, actx)
    for s in range(len(c["Ts"])):
        for pos in range(int(c["ctx"][s]) + int(c["acc"][s]) + 1):
            page, off = int(c["bt"][s, pos // 16]), pos % 16
            np.testing.assert_array_equal(ik[:, page, :, off], ak[:, page, :, off])
            np.testing.assert_array_equal(iv[:, page, :, off], av[:, page, :, off])
            if pos < int(c["ctx"][s]):
                np.testing.assert_array_equal(ik[:, page, :, off], c["kc"][:, page, :, off])


def test_compact_inplace_chain_moves_nothing():
    c = _inplace_case(8)
    for s, T in enumerate(c["Ts"]):
        a = min(T - 1, 5)
        c["path"][s] = -1
        c["path"][s, :a + 1] = np.arange(a + 1)
        c["acc"][s] = a
    pk, pv = O.tree_kv_to_cache(c["kt"], c["vt"], c["kc"], c["vc"], c["bt"], c["ctx"], c["node_off"])
    ik, iv, _, _ = O.kv_compact_inplace(pk, pv, c["bt"], c["ctx"], c["node_off"], c["path"], c["acc"])
    assert np.array_equal(ik, pk) and np.array_equal(iv, pv)


def test_compact_inplace_overlapping_moves_golden():
    """Path 0 -> 2 -> 3 (node 1 rejected): position ctx+1 takes node 2 from
    ctx+2 before ctx+2 takes node 3 from ctx+3; ctx+3 keeps node 3."""
    L, n_kv, d, T, ctx = 1, 1, 2, 4, 14                     # positions 14..17 straddle two pages
    kt = np.arange(T, dtype=np.float64)[None, :, None, None] * np.ones((L, T, n_kv, d))
    kc = np.full((L, 2, n_kv, 16, d), -1.0)
    bt = np.asarray([[1, 0]], np.int32)
    node_off = np.asarray([0, T], np.int32)
    pk, pv = O.tree_kv_to_cache(kt, -kt, kc, kc.copy(), bt, [ctx], node_off)
    path = np.asarray([[0, 2, 3, -1]], np.int32)
    ik, iv, dst, ctx_out = O.kv_compact_inplace(pk, pv, bt, np.asarray([ctx]), node_off, path,
                                                np.asarray([2]))
    def at(a, pos):
        return a[0, bt[0, pos // 16], 0, pos % 16, 0]
    assert [at(ik, ctx + k) for k in range(4)] == [0.0, 2.0, 3.0, 3.0]
    assert [at(iv, ctx + k) for k in range(3)] == [0.0, -2.0, -3.0]
    assert list(dst[0, :3]) == [1 * 16 + 14, 1 * 16 + 15, 0 * 16 + 0]
    assert ctx_out[0] == ctx + 3


# ----------------------------------------------------------------------------
# long reuse drafts: a linear draft verified in place
# ----------------------------------------------------------------------------

def _placed_cache(w):
    kc, vc = O.tree_kv_to_cache(w.k_tree.view(torch.int16).numpy(), w.v_tree.view(torch.int16).numpy(),
                                w.k_cache.view(torch.int16).numpy(), w.v_cache.view(torch.int16).numpy(),
                                w.block_table, w.ctx_len, w.node_off)
    return torch.from_numpy(kc).view(torch.bfloat16), torch.from_numpy(vc).view(torch.bfloat16)


def test_chain_attention_equals_tree_attention_on_chains():
    """Up to 128 nodes a linear draft is a chain tree: in-place chain attention
    equals tree attention over the separate tree arrays."""
    trees = [W.TreeSpec(9, [], [0, 1]), W.TreeSpec(128, [], [0]), W.TreeSpec(1, [], [0])]
    w = W.build("tiny", trees=trees, ctxs=[45, 300, 0])
    kc, vc = _placed_cache(w)
    _, anc = O.tree_prepare(w.parent, w.node_off)
    ref = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0],
                           w.block_table, w.ctx_len, w.node_off, anc)
    out = O.chain_attention(w.q[0], kc[0], vc[0], w.block_table, w.ctx_len, w.node_off)
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


def test_chain_attention_long_draft_is_causal_sdpa():
    """A 300-token draft after a 45-token prefix: torch SDPA (fp64) with the
    causal mask over the whole sequence, every head."""
    T, ctx = 300, 45
    w = W.build("tiny", trees=[W.TreeSpec(T, [], [0, 1])], ctx=ctx)
    kc, vc = _placed_cache(w)
    out = O.chain_attention(w.q[0], kc[0], vc[0], w.block_table, w.ctx_len, w.node_off)
    g = w.n_q // w.n_kv
    keys = torch.stack([_linear_kv(w, 0, 0, hk, range(T), "k") for hk in range(w.n_kv)])
    vals = torch.stack([_linear_kv(w, 0, 0, hk, range(T), "v") for hk in range(w.n_kv)])
    keys = keys.repeat_interleave(g, dim=0)
    vals = vals.repeat_interleave(g, dim=0)
    qq = w.q[0, :T].double().permute(1, 0, 2)
    mask = torch.arange(ctx + T)[None, :] <= (ctx + torch.arange(T))[:, None]
    ref = F.scaled_dot_product_attention(qq[None], keys[None], vals[None], attn_mask=mask)[0]
    np.testing.assert_allclose(out[:T], ref.permute(1, 0, 2).numpy(), rtol=0, atol=1e-12)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_accept_chain_equals_tree_rule_on_chains(seed):
    """accept_chain is accept_path on chain parents, for drafts up to 2048 tokens,
    and a token-by-token replay fixes its length."""
    rng = np.random.default_rng(seed)
    Ts = [1, 2, 300, 2048, 700]
    node_off = np.concatenate([[0], np.cumsum(Ts)]).astype(np.int32)
    total = int(node_off[-1])
    argmax = rng.integers(0, 5, total).astype(np.int32)
    draft = np.empty(total, np.int32)
    parent = np.empty(total, np.int32)
    for s, T in enumerate(Ts):
        o = int(node_off[s])
        stop = int(rng.integers(1, T + 1))              # first rejected position (T: none)
        for i in range(T):
            parent[o + i] = i - 1
            if i == 0:
                draft[o] = 99
            elif i < stop:
                draft[o + i] = argmax[o + i - 1]
            else:
                draft[o + i] = (argmax[o + i - 1] + 1) % 5 if i == stop else int(rng.integers(0, 5))
    acc, path, bonus = O.accept_chain(argmax, draft, node_off)
    acc2, path2, bonus2 = O.accept_path(argmax, draft, parent, node_off)
    np.testing.assert_array_equal(acc, acc2)
    np.testing.assert_array_equal(path, path2)
    np.testing.assert_array_equal(bonus, bonus2)
    for s, T in enumerate(Ts):                            # replay
        o, j = int(node_off[s]), 0
        for k in range(1, T):
            if draft[o + k] != argmax[o + k - 1]:
                break
            j = k
        assert acc[s] == j and bonus[s] == argmax[o + j]


# ----------------------------------------------------------------------------
# Reuse <-> Generate controller
# ----------------------------------------------------------------------------

def test_build_reuse_tree_golden():
    c = np.asarray([5, 6, 7, 8, 5, 6, 9, 1], np.int32)        # "5 6" occurs at 0 and 4
    orig_off = np.asarray([0, len(c)], np.int64)
    mp, nm = O.match_reuse(c, orig_off, np.asarray([[5, 6]]), np.asarray([0]), 4)
    assert list(mp[0, :2]) == [0, 4] and nm[0] == 2
    d, par, off, cpos, gm = O.build_reuse_tree(c, orig_off, mp, nm, [6], 2, 3, 3, gen_tok=[[40, 41]])
    # root, branch 0: c[2..4], branch 1: c[6..7] then past the end, branch 2: none, generated 40 41
    assert list(d) == [6, 7, 8, 5, 9, 1, -1, -1, -1, -1, 40, 41]
    assert list(par) == [-1, 0, 1, 2, 0, 4, 5, 0, 7, 8, 0, 10]
    assert list(cpos) == [1, 2, 3, 4, 6, 7, -1, -1, -1, -1, -1, -1]
    assert list(gm) == [0] * 10 + [1, 1]
    assert list(off) == [0, 12]
    # no match point at all: the root alone holds a token, its position in c is unknown
    c2 = np.asarray([3, 3, 4], np.int32)
    off2 = np.asarray([0, 3], np.int64)
    mp2, nm2 = O.match_reuse(c2, off2, np.asarray([[9, 9]]), np.asarray([0]), 2)
    assert list(mp2[0]) == [-1, -1] and nm2[0] == 0
    d, par, off, cpos, gm = O.build_reuse_tree(c2, off2, mp2, nm2, [9], 2, 2, 2)
    assert list(d) == [9, -1, -1, -1, -1] and list(par) == [-1, 0, 1, 0, 3]
    assert list(cpos) == [-1] * 5 and list(gm) == [0] * 5 and list(off) == [0, 5]


def test_advance_golden():
    out = np.zeros((1, 16), np.int32)
    out[0, :4] = [1, 2, 5, 6]
    d = np.asarray([6, 7, 8, 5, 9, 1, -1, -1, -1, -1, 40, 41], np.int32)
    cpos = np.asarray([1, 2, 3, 4, 6, 7, -1, -1, -1, -1, -1, -1], np.int32)
    path = np.full((1, 12), -1, np.int32)
    path[0, :3] = [0, 1, 2]                                    # accepted 7, 8 (c[2], c[3])
    o2, l2, tail, cur, last = O.advance(out, [4], d, cpos, [0, 12], path, [2], [33], [0], 2)
    assert list(o2[0, :7]) == [1, 2, 5, 6, 7, 8, 33] and l2[0] == 7
    assert list(tail[0]) == [8, 33] and cur[0] == 4 and last[0] == 33    # c[4..] stays the candidate
    path[0, :3] = [0, 10, 11]                                  # the generated branch won
    o3, l3, tail, cur, last = O.advance(out, [4], d, cpos, [0, 12], path, [2], [7], [3], 2)
    assert list(o3[0, :7]) == [1, 2, 5, 6, 40, 41, 7] and cur[0] == 3     # no code consumed


def _depths(parent, node_off):
    dep = np.zeros(len(parent), np.int64)
    for s in range(len(node_off) - 1):
        o = int(node_off[s])
        for i in range(1, int(node_off[s + 1]) - o):
            dep[o + i] = dep[o + int(parent[o + i])] + 1
    return dep


def _edited(rng, c, vocab):
    """c with a replaced span, an inserted span and a deleted span."""
    c = list(c)
    a = int(rng.integers(40, 80))
    c[a:a + 5] = rng.integers(0, vocab, 5).tolist()
    b = int(rng.integers(120, 160))
    c[b:b] = rng.integers(0, vocab, 7).tolist()
    e = int(rng.integers(200, 240))
    del c[e:e + 6]
    return np.asarray(c, np.int32)


@pytest.mark.parametrize("seed,p0,gen", [(0, 20, 0), (1, 35, 3), (2, 8, 4), (3, 60, 2)])
def test_session_reproduces_the_target_text(seed, p0, gen):
    """A whole edit session on the host: match, tree, a synthetic greedy target
    whose next token after k committed tokens is c'[k] (c' = the edited code),
    tree acceptance, commit.  Greedy speculative decoding is lossless, so the
    committed text is c' whatever the drafts; reuse makes it take far fewer
    steps than tokens."""
    rng = np.random.default_rng(seed)
    vocab, n = 1000, 4
    c = rng.integers(0, vocab, 300).astype(np.int32)
    cp = _edited(rng, c, vocab)
    orig_off = np.asarray([0, len(c)], np.int64)
    out = np.zeros((1, len(cp) + 200), np.int32)
    out[0, :p0] = cp[:p0]
    out_len, cursor = np.asarray([p0], np.int32), np.asarray([0], np.int32)
    last = np.asarray([cp[p0 - 1]], np.int32)
    steps = 0
    while out_len[0] < len(cp):
        tail = out[:, out_len[0] - n:out_len[0]]
        mp, nm = O.match_reuse(c, orig_off, tail, cursor, 4)
        proposal = rng.integers(0, vocab, (1, gen)).astype(np.int32) if gen else None
        d, par, off, cpos, _ = O.build_reuse_tree(c, orig_off, mp, nm, last, n, 24, 2, gen_tok=proposal)
        dep = _depths(par, off)
        pos = out_len[0] + dep
        am = np.where(pos < len(cp), cp[np.minimum(pos, len(cp) - 1)], 0).astype(np.int32)
        acc, path, bonus = O.accept_path(am, d, par, off)
        out, out_len, tail, cursor, last = O.advance(out, out_len, d, cpos, off, path, acc, bonus, cursor, n)
        steps += 1
        assert steps < len(cp)
    assert np.array_equal(out[0, :len(cp)], cp)
    assert steps < (len(cp) - p0) // 3
