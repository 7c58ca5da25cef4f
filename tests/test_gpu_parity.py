"""GPU parity: the CUDA verification step, called through the C ABI, against
the fp64 oracle on the same seeded inputs (tolerances in parity_util)."""
import numpy as np
import pytest
import torch

import oracle as O
import parity_util as U
import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    import paper_2506_02780_gb300 as E
    from paper_2506_02780_gb300 import build
    build.build_lib()
    E.lib()


def _E():
    import paper_2506_02780_gb300 as E
    return E


def run_step(w, logits=True, layers=None):
    from paper_2506_02780_gb300 import step as S
    k0, v0 = U.raw16(w.k_cache), U.raw16(w.v_cache)
    st = S.from_workload(w)
    lg = torch.empty((w.total_nodes, w.vocab), dtype=torch.float32, device="cuda") if logits else None
    st.run(logits=lg, layers=layers)
    torch.cuda.synchronize()
    assert _E().ee_read_errors(st.ws) == 0
    return st, lg, k0, v0


def full_check(w, attn_nodes=None, attn_layers=None, lm_nodes=None, logits=True):
    st, lg, k0, v0 = run_step(w, logits=logits)
    U.check_match(w, st)
    anc = U.check_tree(w, st)
    U.check_attention(w, st, range(w.layers) if attn_layers is None else attn_layers, anc,
                      nodes=attn_nodes)
    n_amb = U.check_argmax(w, st, nodes=lm_nodes, logits=lg)
    acc, path = U.check_accept(w, st)
    np.testing.assert_array_equal(acc, w.planted_accept)
    for s in range(w.B):
        assert list(path[s, :acc[s] + 1]) == w.planted_path[s]
    U.check_compact(w, st, k0, v0, acc, path)
    return st, n_amb


# ----------------------------------------------------------------------------
# tiny configuration and edge cases (oracle on every output)
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("seed", [1234, 1, 2])
def test_tiny(seed):
    w = W.build("tiny", seed=seed, device="cuda")
    st, _ = full_check(w)
    assert st.match_pos[0, 0].item() == w.planted_match[0]


def test_tiny_peaky_queries():
    """Large query scale: scores of a few units, exercising the online-softmax rescale."""
    w = W.build("tiny", seed=7, device="cuda", q_std=40.0, ctx=700)
    full_check(w)


def test_exact_ties_pick_lowest_token():
    w = W.build("tiny", seed=8, device="cuda", dup_rows=4)
    st, _ = full_check(w)
    am_ref, cands, lg = O.lm_head_argmax(w.hidden_states, w.lm_w)
    got = st.argmax.cpu().numpy()
    tied = [i for i in range(w.total_nodes) if (lg[i] == lg[i].max()).sum() > 1]
    assert tied
    for i in tied:
        assert got[i] == am_ref[i]           # lowest token id among exact ties


@pytest.mark.parametrize("tree,ctx", [
    (W.TreeSpec(1, [], [0]), 0),                                   # a plain decode step, empty cache
    (W.TreeSpec(1, [], [0]), 16),
    (W.TreeSpec(40, [], W.chain_path(20)), 37),                    # chain only, ragged context
    (W.TreeSpec(1, [(0, 1)] * 15, [0, 5]), 129),                   # star: every node a child of the root
    (W.TreeSpec(100, [(0, 14), (50, 14)], W.chain_path(60)), 1000),  # T = 128, full mask width
    (W.TreeSpec(70, [(3, 20), (3, 20), (69, 10)], [0, 1, 2, 3, 70, 71, 72]), 63),  # path into a branch
])
def test_tree_edge_cases(tree, ctx):
    w = W.build("tiny", seed=11, device="cuda", trees=[tree], ctx=ctx)
    full_check(w)


def test_multi_sequence_small():
    w = W.build("batched", seed=21, device="cuda", layers=2, vocab=8192, hidden=512)
    full_check(w)


def test_repeat_runs_bit_identical():
    w = W.build("tiny", seed=5, device="cuda")
    from paper_2506_02780_gb300 import step as S
    st = S.from_workload(w)
    outs = []
    for _ in range(5):
        st.run()
        torch.cuda.synchronize()
        outs.append([t.clone() for t in (st.match_pos, st.argmax, st.path, st.accept_len, st.bonus,
                                         st.dst_slot, st.attn_out)])
    for o in outs[1:]:
        for a, b in zip(outs[0], o):
            assert torch.equal(a, b)


# ----------------------------------------------------------------------------
# balanced attention launch (one CTA per SM, an equal share of all row blocks'
# tiles, row blocks split across CTAs and merged through counters)
# ----------------------------------------------------------------------------

_RAGGED = [W.TreeSpec(100, [(0, 14), (50, 14)], W.chain_path(60)),   # T = 128
           W.TreeSpec(1, [], [0]),                                    # a decode step
           W.TreeSpec(60, [(10, 17)], W.chain_path(30)),              # T = 77
           W.TreeSpec(100, [(3, 28)], [0, 1, 2, 3, 100, 101, 102]),   # T = 128, path into a branch
           W.TreeSpec(40, [], W.chain_path(20))]                      # T = 40


@pytest.mark.parametrize("ctxs", [
    [5000, 0, 3001, 4500, 17],      # ragged; an empty cache; a one-page context
    [4999, 4096, 1, 127, 2049],
])
def test_balanced_ragged(ctxs):
    """Five sequences of 1 to 128 nodes over ragged contexts with 6 query heads
    per KV head: 60 row blocks leave a quarter of the SMs idle in an equal-chunk
    launch, so the planner picks the balanced launch; CTAs' shares cross row
    blocks, whole small row blocks sit inside one CTA, and large ones are split
    over several CTAs.  Every node and head is checked against the oracle."""
    E = _E()
    w = W.build("tiny", seed=31, device="cuda", trees=_RAGGED, ctxs=ctxs, n_q=12, n_kv=2)
    plan = E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, int(w.ctx_len.max()))
    assert plan["mode"] == "balanced", plan
    full_check(w)


def test_balanced_many_pieces():
    """One sequence, 8 KV heads x 5 row blocks of 158 tiles: each row block is
    split over 4 to 5 CTAs (sampled nodes, every head)."""
    E = _E()
    w = W.build("tiny", seed=32, device="cuda", trees=[_RAGGED[0]], ctx=20000, n_q=40, n_kv=8)
    plan = E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, int(w.ctx_len.max()))
    assert plan["mode"] == "balanced", plan
    full_check(w, attn_nodes=_sample_nodes(w, 12, 3))


def test_balanced_repeat_bit_identical():
    """The merge order of a split row block is fixed (piece order), so repeated
    balanced launches give identical outputs, and the counters return to zero."""
    E = _E()
    from paper_2506_02780_gb300 import step as S
    w = W.build("tiny", seed=33, device="cuda", trees=_RAGGED, ctxs=[5000, 0, 3001, 4500, 17],
                n_q=12, n_kv=2)
    st = S.from_workload(w)
    assert E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, st.max_ctx)["mode"] == "balanced"
    outs = []
    for _ in range(8):
        st.run()
        torch.cuda.synchronize()
        outs.append(st.attn_out.clone())
    assert E.ee_read_errors(st.ws) == 0
    for o in outs[1:]:
        assert torch.equal(outs[0], o)


def test_launch_plans_of_the_configurations():
    """The plans the configurations are timed with: 7b fills 144 SMs with 9
    equal chunks of 16 row blocks; 33b (56 row blocks of 257 tiles) and the
    ragged batch take the balanced launch."""
    E = _E()
    p7 = E.ee_attn_plan(1, 64, 28, 4, 4096)
    assert p7["mode"] == "cooperative" and p7["splits"] == 9 and p7["ctas"] == 144, p7
    p33 = E.ee_attn_plan(1, 128, 56, 8, 32768)
    assert p33["mode"] == "balanced", p33
    pb = E.ee_attn_plan(8, 96, 28, 4, 16384)
    assert pb["mode"] == "balanced", pb


# ----------------------------------------------------------------------------
# device-detected bad input: error word set, access skipped, context usable
# ----------------------------------------------------------------------------

def test_device_error_word():
    E = _E()
    from paper_2506_02780_gb300 import step as S
    w = W.build("tiny", seed=3, device="cuda")
    st = S.from_workload(w)
    st.inp["block_table"][0, 1] = w.num_pages + 5            # out-of-range page inside the context
    st.run()
    bits = E.ee_read_errors(st.ws)
    assert bits & 0x04
    st.inp["block_table"][0, 1] = int(w.block_table[0, 1])
    st.inp["cursor"][0] = -1
    st.run()
    assert E.ee_read_errors(st.ws) & 0x01
    st.inp["cursor"][0] = int(w.cursor[0])
    bad_parent = st.inp["parent"].clone()
    st.inp["parent"][3] = 7                                   # parent after child
    st.run()
    assert E.ee_read_errors(st.ws) & 0x02
    st.inp["parent"].copy_(bad_parent)
    E.ee_workspace_init(st.ws)
    st.run()                                                  # a clean call afterwards works
    torch.cuda.synchronize()
    assert E.ee_read_errors(st.ws) == 0
    U.check_accept(w, st)


def test_attention_plans_within_a_small_workspace():
    """A workspace with no room for partial slots (sized for an empty context)
    runs the plan that needs none -- one CTA per row block over its whole
    context -- and still matches the oracle; below the fixed head the call is
    refused before anything is launched."""
    E = _E()
    from paper_2506_02780_gb300 import step as S
    w = W.build("tiny", seed=4, device="cuda")
    st = S.from_workload(w)
    small = E.new_workspace(w.B, w.total_nodes, w.n_q, 0)
    assert small.numel() < st.ws.numel()
    x = st.inp
    anc = O.tree_prepare(w.parent, w.node_off)[1]
    anc_d = torch.from_numpy(anc.view(np.int64)).cuda()
    out = torch.full_like(st.attn_out[0], 7.0)
    E.ee_tree_verify_attn(x["q"][0], x["k_tree"][0], x["v_tree"][0], x["k_cache"][0], x["v_cache"][0],
                          x["block_table"], x["ctx_len"], st.max_ctx, x["node_off"], anc_d, st.max_T, st.scale,
                          out, small)
    torch.cuda.synchronize()
    assert E.ee_read_errors(small) == 0
    ref = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0], w.block_table,
                           w.ctx_len, w.node_off, anc)
    U.assert_close(out.cpu().numpy(), ref, "attention, one-chunk plan")
    tiny_ws = small[:1024]
    out.fill_(7.0)
    with pytest.raises(E.EEError) as ei:
        E.ee_tree_verify_attn(x["q"][0], x["k_tree"][0], x["v_tree"][0], x["k_cache"][0], x["v_cache"][0],
                              x["block_table"], x["ctx_len"], st.max_ctx, x["node_off"], anc_d, st.max_T,
                              st.scale, out, tiny_ws)
    assert ei.value.status == 5
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())


# ----------------------------------------------------------------------------
# full-size configurations (sampled attention outputs, launch configuration as timed)
# ----------------------------------------------------------------------------

def _sample_nodes(w, k, seed=0):
    rng = np.random.default_rng(seed)
    nodes = set(rng.choice(w.total_nodes, size=min(k, w.total_nodes), replace=False).tolist())
    for s in range(w.B):                       # first and last node of every tree
        nodes.add(int(w.node_off[s]))
        nodes.add(int(w.node_off[s + 1]) - 1)
    return sorted(nodes)


@pytest.mark.slow
def test_7b_full_size():
    w = W.build("7b", device="cuda")
    full_check(w, attn_nodes=_sample_nodes(w, 10), logits=False)


@pytest.mark.slow
def test_batched_full_size():
    w = W.build("batched", device="cuda")
    lm_nodes = sorted(set(_sample_nodes(w, 40, 1)) |
                      {int(w.node_off[s]) + u for s in range(w.B) for u in w.planted_path[s]})
    full_check(w, attn_nodes=_sample_nodes(w, 24), attn_layers=[0, 13, 27], lm_nodes=lm_nodes,
               logits=False)


@pytest.mark.slow
def test_33b_full_size():
    w = W.build("33b", device="cuda")
    full_check(w, attn_nodes=_sample_nodes(w, 6), attn_layers=[0, 61], logits=False)


@pytest.mark.parametrize("n", [2, 4, 8])
def test_sweep_match_full_size(n):
    E = _E()
    w = W.build("sweep", device="cuda", n=n, layers=1, seed=1238 + n)
    dev = "cuda"
    i32 = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    mp = torch.empty((w.B, 16), dtype=torch.int32, device=dev)
    nm = torch.empty(w.B, dtype=torch.int32, device=dev)
    ws = E.new_workspace(w.B, w.total_nodes, 1, 0)
    E.ee_match_reuse(i32(w.orig_tokens), torch.as_tensor(w.orig_off, device=dev), i32(w.tail),
                     i32(w.cursor), 16, mp, nm, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    pos, cnt = O.match_reuse(w.orig_tokens, w.orig_off, w.tail, w.cursor, 16)
    np.testing.assert_array_equal(mp.cpu().numpy(), pos)
    np.testing.assert_array_equal(nm.cpu().numpy(), cnt)
    assert (cnt > 1).any()                    # repeated segments make some tails ambiguous


@pytest.mark.parametrize("max_matches", [1, 16, 1024])
def test_match_split_ranges(max_matches):
    """Codes long enough for several CTAs per sequence (the scan is split into
    ranges whose hits are concatenated by the last CTA to finish): hits planted
    every 2,999 positions, none at all, dense (every 7th position, more than
    1,024 hits), only before the cursor, and in a code shorter than one range;
    positions and counts equal the oracle's.  The same inputs with a workspace
    of only the fixed head (one CTA per sequence) give the same result."""
    E = _E()
    rng = np.random.default_rng(5)
    n = 3
    pat = np.array([1001, 1002, 1003], np.int32)            # tokens of c are drawn below 1000
    lens = [65536, 20000, 40000, 30000, 100]
    codes = []
    for s, ln in enumerate(lens):
        c = rng.integers(0, 1000, ln).astype(np.int32)
        step = {0: 2999, 2: 7, 3: 1000, 4: 50}.get(s)
        if step:
            for p0 in range(5, ln - n - 1, step):
                if s == 3 and p0 > 10000:
                    break
                c[p0:p0 + n] = pat
        codes.append(c)
    orig = np.concatenate(codes)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tail = np.tile(pat, (len(lens), 1))
    cursor = np.array([17, 0, 3, 12000, 0], np.int32)
    pos, cnt = O.match_reuse(orig, off, tail, cursor, max_matches)
    assert cnt[2] > 1024 and cnt[1] == 0 and cnt[3] == 0 and cnt[0] > 16
    dev = "cuda"
    args = (torch.as_tensor(orig, device=dev), torch.as_tensor(off, device=dev),
            torch.as_tensor(tail, device=dev), torch.as_tensor(cursor, device=dev))
    head = E.lib().ee_workspace_size(len(lens), 1, 1, 128, 0)
    for ws in (E.new_workspace(len(lens), 64, 1, 0), torch.zeros(16896, dtype=torch.uint8, device=dev)):
        for _ in range(2):                                   # the tickets are back at zero
            mp = torch.full((len(lens), max_matches), 7, dtype=torch.int32, device=dev)
            nm = torch.full((len(lens),), 7, dtype=torch.int32, device=dev)
            E.ee_match_reuse(*args, max_matches, mp, nm, ws)
            torch.cuda.synchronize()
            assert E.ee_read_errors(ws) == 0
            np.testing.assert_array_equal(mp.cpu().numpy(), pos)
            np.testing.assert_array_equal(nm.cpu().numpy(), cnt)
    assert head > 16896


def test_sweep_compaction_full_size():
    E = _E()
    w = W.build("sweep", device="cuda")
    dev = "cuda"
    i32 = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    path = np.full((w.B, w.max_T), -1, np.int32)
    for s in range(w.B):
        path[s, :len(w.planted_path[s])] = w.planted_path[s]
    k0, v0 = U.raw16(w.k_cache), U.raw16(w.v_cache)
    ctx_out = torch.empty(w.B, dtype=torch.int32, device=dev)
    dst = torch.empty((w.B, w.max_T), dtype=torch.int32, device=dev)
    ws = E.new_workspace(w.B, w.total_nodes, 1, 0)
    E.ee_kv_compact(w.k_tree, w.v_tree, w.k_cache, w.v_cache, i32(w.block_table), i32(w.ctx_len),
                    ctx_out, i32(w.node_off), i32(path), i32(w.planted_accept), dst, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    kc, vc, dref, cref = O.kv_compact(U.raw16(w.k_tree), U.raw16(w.v_tree), k0, v0, w.block_table,
                                      w.ctx_len, w.node_off, path, w.planted_accept)
    np.testing.assert_array_equal(dst.cpu().numpy(), dref)
    np.testing.assert_array_equal(ctx_out.cpu().numpy(), cref)
    assert np.array_equal(U.raw16(w.k_cache), kc) and np.array_equal(U.raw16(w.v_cache), vc)


@pytest.mark.parametrize("n_kv,n_q,layers", [(1, 8, 1), (3, 21, 5), (8, 56, 6), (2, 8, 4)])
def test_compaction_head_counts_and_layer_groups(n_kv, n_q, layers):
    """The compaction kernel's instances: KV head counts with a compiled-in
    count (1, 2, 8) and the generic one (3); layer counts that fill the groups of
    four exactly (4), leave a remainder (5, 6) or one layer.  Cache bytes, slots
    and new context lengths bit-exact against the oracle's sequential append."""
    E = _E()
    w = W.build("sweep", B=6, layers=layers, n_kv=n_kv, n_q=n_q, seed=40 + n_kv)
    dev = "cuda"
    i32 = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    path = np.full((w.B, w.max_T), -1, np.int32)
    for s in range(w.B):
        path[s, :len(w.planted_path[s])] = w.planted_path[s]
    k0, v0 = U.raw16(w.k_cache), U.raw16(w.v_cache)
    kc_d = w.k_cache.to(dev)
    vc_d = w.v_cache.to(dev)
    ctx_out = torch.empty(w.B, dtype=torch.int32, device=dev)
    dst = torch.empty((w.B, w.max_T), dtype=torch.int32, device=dev)
    ws = E.new_workspace(w.B, w.total_nodes, 1, 0)
    E.ee_kv_compact(w.k_tree.to(dev), w.v_tree.to(dev), kc_d, vc_d, i32(w.block_table), i32(w.ctx_len),
                    ctx_out, i32(w.node_off), i32(path), i32(w.planted_accept), dst, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    kc, vc, dref, cref = O.kv_compact(U.raw16(w.k_tree), U.raw16(w.v_tree), k0, v0, w.block_table,
                                      w.ctx_len, w.node_off, path, w.planted_accept)
    np.testing.assert_array_equal(dst.cpu().numpy(), dref)
    np.testing.assert_array_equal(ctx_out.cpu().numpy(), cref)
    assert np.array_equal(U.raw16(kc_d), kc) and np.array_equal(U.raw16(vc_d), vc)


@pytest.mark.parametrize("n", [9, 32])
def test_match_long_ngrams_split(n):
    """n-grams longer than the vectorised compare covers (the general loop),
    over codes split across several CTAs per sequence: hits planted every 1,777
    positions, including across range and tile boundaries."""
    E = _E()
    rng = np.random.default_rng(n)
    pat = (2000 + np.arange(n)).astype(np.int32)
    lens = [65536, 50000, 9000, 70000]
    codes = []
    for ln in lens:
        c = rng.integers(0, 2000, ln).astype(np.int32)
        for p0 in range(3, ln - n - 1, 1777):
            c[p0:p0 + n] = pat
        codes.append(c)
    orig = np.concatenate(codes)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tail = np.tile(pat, (len(lens), 1))
    cursor = np.array([0, 4000, 8999 - n, 1], np.int32)
    pos, cnt = O.match_reuse(orig, off, tail, cursor, 64)
    dev = "cuda"
    mp = torch.empty((len(lens), 64), dtype=torch.int32, device=dev)
    nm = torch.empty(len(lens), dtype=torch.int32, device=dev)
    ws = E.new_workspace(len(lens), 64, 1, 0)
    E.ee_match_reuse(torch.as_tensor(orig, device=dev), torch.as_tensor(off, device=dev),
                     torch.as_tensor(tail, device=dev), torch.as_tensor(cursor, device=dev), 64, mp, nm, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    np.testing.assert_array_equal(mp.cpu().numpy(), pos)
    np.testing.assert_array_equal(nm.cpu().numpy(), cnt)
    assert cnt[0] > 30


def test_match_bad_sequences_in_a_split_batch():
    """A batch whose long codes are split over several CTAs, with one sequence
    whose offsets decrease and one with a negative cursor: the device error
    word reports EE_DEVERR_MATCH_ARGS, those sequences report no match, and the
    others equal the oracle's -- on two calls in a row (the tickets of the
    split sequences return to zero; the bad ones take none)."""
    E = _E()
    rng = np.random.default_rng(8)
    n = 4
    pat = np.array([900, 901, 902, 903], np.int32)
    lens = [60000, 30000, 50000, 20000]
    codes = []
    for ln in lens:
        c = rng.integers(0, 800, ln).astype(np.int32)
        for p0 in range(11, ln - n - 1, 997):
            c[p0:p0 + n] = pat
        codes.append(c)
    orig = np.concatenate(codes)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    bad_off = off.copy()
    bad_off[2] = bad_off[1] - 5               # sequence 1: end before start
    cursor = np.array([0, 0, 0, -3], np.int32)  # sequence 3: negative cursor
    tail = np.tile(pat, (len(lens), 1))
    good = [0, 2]                               # sequence 2 spans [bad_off[2], off[3])
    exp = {s: O.match_reuse(orig, bad_off[s:s + 2] - 0, tail[s:s + 1], cursor[s:s + 1], 16) for s in good}
    dev = "cuda"
    ws = E.new_workspace(len(lens), 64, 1, 0)
    for _ in range(2):
        mp = torch.full((len(lens), 16), 7, dtype=torch.int32, device=dev)
        nm = torch.full((len(lens),), 7, dtype=torch.int32, device=dev)
        E.ee_match_reuse(torch.as_tensor(orig, device=dev), torch.as_tensor(bad_off, device=dev),
                         torch.as_tensor(tail, device=dev), torch.as_tensor(cursor, device=dev), 16, mp, nm, ws)
        torch.cuda.synchronize()
        assert E.ee_read_errors(ws) == 0x01
        got_p, got_n = mp.cpu().numpy(), nm.cpu().numpy()
        for s in good:
            np.testing.assert_array_equal(got_p[s], exp[s][0][0])
            assert got_n[s] == exp[s][1][0] > 16
        for s in (1, 3):
            assert got_n[s] == 0 and (got_p[s] == -1).all()


def test_split_row_block_counts_shared_by_plans():
    """A workspace shared by launches with different plans (cooperative chunks
    with different chunk counts, a balanced launch) keeps every result exact:
    the row blocks' arrival counts are never reset, every launch raises them by
    the same constant, so a count left by a 9-piece plan is a valid start for a
    5-piece one.  Each call is bit-identical to the same call on a fresh
    workspace, and close to the oracle."""
    E = _E()
    from paper_2506_02780_gb300 import step as S
    cases = [W.build("tiny", seed=51, device="cuda", ctx=6000),
             W.build("tiny", seed=52, device="cuda", ctx=1500),
             W.build("tiny", seed=53, device="cuda", trees=_RAGGED, ctxs=[5000, 0, 3001, 4500, 17],
                     n_q=12, n_kv=2)]
    steps = [S.from_workload(w) for w in cases]
    plans = [E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, st.max_ctx) for w, st in zip(cases, steps)]
    assert len({(p["mode"], p["splits"]) for p in plans}) == 3, plans
    shared = E.new_workspace(5, max(w.total_nodes for w in cases), 12, 6000)
    ref = []
    for w, st in zip(cases, steps):                # fresh workspaces: the reference outputs
        st.run()
        torch.cuda.synchronize()
        assert E.ee_read_errors(st.ws) == 0
        ref.append(st.attn_out.clone())
    anc = [U.check_tree(w, st) for w, st in zip(cases, steps)]
    for rnd in range(3):
        for i, (w, st) in enumerate(zip(cases, steps)):
            x = st.inp
            out = torch.full_like(st.attn_out[0], float("nan"))
            E.ee_tree_verify_attn(x["q"][0], x["k_tree"][0], x["v_tree"][0], x["k_cache"][0], x["v_cache"][0],
                                  x["block_table"], x["ctx_len"], st.max_ctx, x["node_off"], st.anc, st.max_T,
                                  st.scale, out, shared)
            torch.cuda.synchronize()
            assert E.ee_read_errors(shared) == 0, (rnd, i)
            assert torch.equal(out, ref[i][0]), (rnd, i, plans[i])
    for i, (w, st) in enumerate(zip(cases, steps)):
        U.check_attention(w, st, [0], anc[i], nodes=_sample_nodes(w, 12, 3))


@pytest.mark.parametrize("v_scale_log2", [24, -40])
def test_split_values_far_from_unit_scale(v_scale_log2):
    """Split row blocks hand partial (O, max, sum) over through the workspace and
    merge them: values far above fp16's largest (2^24 times N(0, 1) / 11) and far
    below its smallest normal (2^-40 times that) come out with the oracle's
    relative accuracy, i.e. nothing on the way narrows the fp32 range.  The
    values are scaled by an exact power of two, so the oracle sees the same bf16
    inputs."""
    E = _E()
    from paper_2506_02780_gb300 import step as S
    f = 2.0 ** v_scale_log2
    w = W.build("tiny", seed=61, device="cuda", trees=_RAGGED, ctxs=[5000, 0, 3001, 4500, 17], n_q=12, n_kv=2)
    w.v_cache.mul_(f)
    w.v_tree.mul_(f)
    st = S.from_workload(w)
    plan = E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, st.max_ctx)
    assert plan["splits"] > 1 or plan["mode"] == 3, plan   # partials are merged
    st.run()
    torch.cuda.synchronize()
    assert E.ee_read_errors(st.ws) == 0
    anc = U.check_tree(w, st)
    nodes = _sample_nodes(w, 16, 5)
    ref = O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0], w.block_table,
                           w.ctx_len, w.node_off, anc, nodes=nodes)[nodes]
    got = st.attn_out[0].cpu().double().numpy()[nodes]
    assert np.isfinite(got).all()
    U.assert_close(got / f, ref / f, f"attention, values scaled by 2^{v_scale_log2}")
