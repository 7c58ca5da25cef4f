"""GPU parity of in-place speculative K/V: the tree's K/V sit in the cache at
positions ctx + i (placed by the oracle), ee_tree_verify_attn_inplace attends
over them and ee_kv_compact_inplace moves the accepted path down.  Attention is
checked against the oracle's tree attention over the original tree arrays
(tolerances in parity_util); the compacted cache, slots and new context
lengths bit-exactly against the oracle's kv_compact_inplace."""
import math

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


def _inputs(w):
    """Device inputs: the cache with the tree's K/V placed at ctx + i (oracle,
    on the host), a block table padded so that max_ctx + max_T positions have
    columns, the ancestor masks."""
    kc, vc = O.tree_kv_to_cache(U.raw16(w.k_tree), U.raw16(w.v_tree), U.raw16(w.k_cache),
                                U.raw16(w.v_cache), w.block_table, w.ctx_len, w.node_off)
    max_ctx = int(w.ctx_len.max())
    cols = max(w.block_table.shape[1], math.ceil((max_ctx + w.max_T) / 16))
    bt = np.full((w.B, cols), -1, np.int32)
    bt[:, :w.block_table.shape[1]] = w.block_table
    _, anc = O.tree_prepare(w.parent, w.node_off)
    dev = torch.device("cuda")
    return dict(
        kc_np=kc, vc_np=vc,
        kc=torch.from_numpy(kc).view(torch.bfloat16).to(dev),
        vc=torch.from_numpy(vc).view(torch.bfloat16).to(dev),
        bt=torch.from_numpy(bt).to(dev),
        ctx=torch.as_tensor(w.ctx_len, dtype=torch.int32, device=dev),
        node_off=torch.as_tensor(w.node_off, dtype=torch.int32, device=dev),
        anc=torch.from_numpy(anc.view(np.int64)).to(dev),
        anc_np=anc, max_ctx=max_ctx)


def check_inplace(w, layers=None, nodes=None, expect_mode=None):
    E = _E()
    x = _inputs(w)
    if expect_mode is not None:
        plan = E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, x["max_ctx"], inplace=True)
        assert plan["mode"] == expect_mode, plan
    ws = E.new_workspace(w.B, w.total_nodes, w.n_q, x["max_ctx"])
    scale = 1.0 / math.sqrt(128)
    for l in (range(w.layers) if layers is None else layers):
        out = torch.full((w.total_nodes, w.n_q, 128), float("nan"), dtype=torch.float32, device="cuda")
        E.ee_tree_verify_attn_inplace(w.q[l], x["kc"][l], x["vc"][l], x["bt"], x["ctx"], x["max_ctx"],
                                      x["node_off"], x["anc"], w.max_T, scale, out, ws)
        torch.cuda.synchronize()
        assert E.ee_read_errors(ws) == 0
        ref = O.tree_attention(w.q[l], w.k_tree[l], w.v_tree[l], w.k_cache[l], w.v_cache[l], w.block_table,
                               w.ctx_len, w.node_off, x["anc_np"], nodes=nodes)
        U.assert_close(out.cpu().numpy(), ref, f"in-place attention layer {l}")
    # compaction of the planted path
    path = np.full((w.B, w.max_T), -1, np.int32)
    for s in range(w.B):
        path[s, :len(w.planted_path[s])] = w.planted_path[s]
    acc = np.asarray(w.planted_accept, np.int32)
    ctx_out = torch.zeros(w.B, dtype=torch.int32, device="cuda")
    dst = torch.full((w.B, w.max_T), 7, dtype=torch.int32, device="cuda")
    E.ee_kv_compact_inplace(x["kc"], x["vc"], x["bt"], x["ctx"], ctx_out, x["node_off"],
                            torch.from_numpy(path).cuda(), torch.from_numpy(acc).cuda(), w.total_nodes, dst, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    rk, rv, rdst, rctx = O.kv_compact_inplace(x["kc_np"], x["vc_np"], w.block_table, w.ctx_len, w.node_off,
                                              path, acc)
    np.testing.assert_array_equal(dst.cpu().numpy(), rdst)
    np.testing.assert_array_equal(ctx_out.cpu().numpy(), rctx)
    assert np.array_equal(U.raw16(x["kc"]), rk), "compacted K cache"
    assert np.array_equal(U.raw16(x["vc"]), rv), "compacted V cache"
    moved = sum(int((path[s, :acc[s] + 1] != np.arange(acc[s] + 1)).sum()) for s in range(w.B))
    return moved


@pytest.mark.parametrize("tree,ctx", [
    (W.TreeSpec(1, [], [0]), 0),                                   # a decode step, empty cache
    (W.TreeSpec(12, [(0, 4)], W.chain_path(7)), 512),              # the tiny configuration's tree
    (W.TreeSpec(40, [], W.chain_path(20)), 37),                    # ragged context: tree mid-page
    (W.TreeSpec(1, [(0, 1)] * 15, [0, 5]), 129),                   # star: a move from node 5
    (W.TreeSpec(100, [(0, 14), (50, 14)], W.chain_path(60)), 1000),  # T = 128
    (W.TreeSpec(70, [(3, 20), (3, 20), (69, 10)], [0, 1, 2, 3, 70, 71, 72]), 63),  # path into a branch
    (W.TreeSpec(100, [(3, 28)], [0, 1, 2, 3, 100, 101, 102]), 4000),  # T = 128 across a tile edge
])
def test_inplace_edge_cases(tree, ctx):
    w = W.build("tiny", seed=41, device="cuda", trees=[tree], ctx=ctx)
    check_inplace(w)


def test_inplace_branch_paths_move():
    """Every sequence's accepted path leaves the chain: the compaction moves."""
    trees = [W.TreeSpec(30, [(5, 10)], [0, 1, 2, 3, 4, 5, 30, 31, 32]),
             W.TreeSpec(8, [(0, 6), (2, 5)], [0, 8, 9, 10]),
             W.TreeSpec(64, [(10, 30)], [0] + list(range(1, 11)) + list(range(64, 80)))]
    w = W.build("tiny", seed=42, device="cuda", trees=trees, ctxs=[300, 17, 2047])
    assert check_inplace(w) > 0


_RAGGED = [W.TreeSpec(100, [(0, 14), (50, 14)], W.chain_path(60)),
           W.TreeSpec(1, [], [0]),
           W.TreeSpec(60, [(10, 17)], W.chain_path(30)),
           W.TreeSpec(100, [(3, 28)], [0, 1, 2, 3, 100, 101, 102]),
           W.TreeSpec(40, [], W.chain_path(20))]


@pytest.mark.parametrize("ctxs", [[5000, 0, 3001, 4500, 17], [4999, 4096, 1, 127, 2049]])
def test_inplace_balanced_ragged(ctxs):
    """The balanced launch over in-place trees (every node, every head)."""
    w = W.build("tiny", seed=43, device="cuda", trees=_RAGGED, ctxs=ctxs, n_q=12, n_kv=2)
    check_inplace(w, expect_mode="balanced")


def test_inplace_multi_sequence():
    w = W.build("batched", seed=44, device="cuda", layers=2, vocab=8192, hidden=512)
    check_inplace(w)


@pytest.mark.slow
def test_inplace_7b_full_size():
    """The 7b workload's shapes and launch plan (sampled attention nodes)."""
    w = W.build("7b", device="cuda", layers=2)
    rng = np.random.default_rng(0)
    nodes = sorted(set(rng.choice(w.total_nodes, 10, replace=False).tolist()) | {0, w.total_nodes - 1})
    assert check_inplace(w, nodes=nodes, expect_mode="cooperative") == 0   # the planted path is the chain


@pytest.mark.parametrize("name,kw", [("tiny", {}),
                                     ("batched", dict(layers=2, vocab=8192, hidden=512))])
def test_step_inplace_kv(name, kw):
    """VerifyStep with inplace_kv: set-up places the tree's K/V in the cache;
    the step's attention, acceptance and compaction match the oracle."""
    E = _E()
    from paper_2506_02780_gb300 import step as S
    w = W.build(name, seed=45, device="cuda", **kw)
    st = S.from_workload(w, inplace_kv=True)
    kc0, vc0 = U.raw16(w.k_cache), U.raw16(w.v_cache)     # after placement, before the step
    ref_k, ref_v = O.tree_kv_to_cache(U.raw16(w.k_tree), U.raw16(w.v_tree), kc0, vc0, w.block_table,
                                      w.ctx_len, w.node_off)
    assert np.array_equal(kc0, ref_k) and np.array_equal(vc0, ref_v)   # placement as the oracle places
    st.run()
    torch.cuda.synchronize()
    assert E.ee_read_errors(st.ws) == 0
    anc = U.check_tree(w, st)
    U.check_attention(w, st, range(w.layers), anc)
    acc, path = U.check_accept(w, st)
    rk, rv, rdst, rctx = O.kv_compact_inplace(kc0, vc0, w.block_table, w.ctx_len, w.node_off, path, acc)
    np.testing.assert_array_equal(st.dst_slot.cpu().numpy(), rdst)
    np.testing.assert_array_equal(st.ctx_out.cpu().numpy(), rctx)
    assert np.array_equal(U.raw16(w.k_cache), rk) and np.array_equal(U.raw16(w.v_cache), rv)


@pytest.mark.parametrize("inplace", [False, True])
def test_compaction_waits_for_the_lm_head(inplace):
    """The compaction starts before the LM head has finished (programmatic
    dependent launch) and must read path / accept_len only after its wait.  The
    outputs are poisoned before every step, and later calls in one process
    overlap the launches: a premature read shows as a device error or a wrong
    new context length."""
    E = _E()
    from paper_2506_02780_gb300 import step as S
    w = W.build("batched", seed=45, device="cuda", layers=2, vocab=8192, hidden=512)
    st = S.from_workload(w, inplace_kv=inplace)
    want = None
    for _ in range(4):
        st.accept_len.fill_(-7)
        st.path.fill_(-7)
        st.ctx_out.fill_(-5)
        st.run()
        torch.cuda.synchronize()
        assert E.ee_read_errors(st.ws) == 0
        got = st.ctx_out.cpu().numpy()
        np.testing.assert_array_equal(got, w.ctx_len + st.accept_len.cpu().numpy() + 1)
        want = got if want is None else want
        np.testing.assert_array_equal(got, want)
