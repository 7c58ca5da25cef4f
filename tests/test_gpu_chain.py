"""GPU parity of long reuse drafts: linear drafts of up to 2048 tokens verified
in place.  Their K/V are placed in the cache at positions ctx + i by the oracle;
ee_chain_verify_attn is checked against the oracle's causal chain attention
(tolerances in parity_util), ee_lmhead_accept with anc NULL against the
longest-prefix rule, and both compactions bit-exactly."""
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


def _placed(w):
    """The cache with every draft's K/V at ctx + i (oracle, on the host) and a
    block table with a column for every position below max_ctx + max_T."""
    kc, vc = O.tree_kv_to_cache(U.raw16(w.k_tree), U.raw16(w.v_tree), U.raw16(w.k_cache),
                                U.raw16(w.v_cache), w.block_table, w.ctx_len, w.node_off)
    max_ctx = int(w.ctx_len.max())
    cols = max(w.block_table.shape[1], math.ceil((max_ctx + w.max_T) / 16))
    bt = np.full((w.B, cols), -1, np.int32)
    bt[:, :w.block_table.shape[1]] = w.block_table
    dev = torch.device("cuda")
    return dict(kc_np=kc, vc_np=vc, kc=torch.from_numpy(kc).view(torch.bfloat16).to(dev),
                vc=torch.from_numpy(vc).view(torch.bfloat16).to(dev), bt=torch.from_numpy(bt).to(dev),
                ctx=torch.as_tensor(w.ctx_len, dtype=torch.int32, device=dev),
                node_off=torch.as_tensor(w.node_off, dtype=torch.int32, device=dev), max_ctx=max_ctx)


def check_chain_attention(w, nodes=None, layers=(0,)):
    E = _E()
    x = _placed(w)
    ws = E.new_workspace(w.B, w.total_nodes, w.n_q, x["max_ctx"])
    plan = E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, x["max_ctx"], inplace="chain")
    for l in layers:
        out = torch.full((w.total_nodes, w.n_q, 128), float("nan"), dtype=torch.float32, device="cuda")
        E.ee_chain_verify_attn(w.q[l], x["kc"][l], x["vc"][l], x["bt"], x["ctx"], x["max_ctx"], x["node_off"],
                               w.max_T, 1.0 / math.sqrt(128), out, ws)
        torch.cuda.synchronize()
        assert E.ee_read_errors(ws) == 0
        kc = torch.from_numpy(x["kc_np"][l]).view(torch.bfloat16)
        vc = torch.from_numpy(x["vc_np"][l]).view(torch.bfloat16)
        ref = O.chain_attention(w.q[l], kc, vc, w.block_table, w.ctx_len, w.node_off, nodes=nodes)
        U.assert_close(out.cpu().numpy(), ref, f"chain attention layer {l}")
    return plan


_SMALL = dict(layers=1, vocab=8192, hidden=512, n_q=8, n_kv=2)


@pytest.mark.parametrize("trees,ctxs", [
    ([W.TreeSpec(1000, [], W.chain_path(999)), W.TreeSpec(1, [], [0]), W.TreeSpec(300, [], W.chain_path(17))],
     [37, 0, 2000]),
    ([W.TreeSpec(2048, [], W.chain_path(1500))], [4096]),
    ([W.TreeSpec(129, [], W.chain_path(5)), W.TreeSpec(640, [], W.chain_path(639))], [127, 1]),
])
def test_chain_attention_every_node(trees, ctxs):
    """Ragged linear drafts (1 to 2048 tokens, contexts 0 to 4096): every node
    and head against the oracle."""
    w = W.build("long", seed=51, device="cuda", trees=trees, ctxs=ctxs, **_SMALL)
    check_chain_attention(w)


def test_chain_attention_7b_heads_sampled():
    """The long workload with the 7B-coder heads (28 / 4): sampled nodes
    spanning every row block's first and last rows."""
    w = W.build("long", seed=52, device="cuda", layers=1, vocab=8192, hidden=512)
    g = w.n_q // w.n_kv
    rng = np.random.default_rng(0)
    nodes = set(rng.choice(w.total_nodes, 12, replace=False).tolist()) | {0, w.total_nodes - 1}
    for rb in (0, 1, 55, 111):                       # nodes at row-block edges
        nodes |= {min(w.total_nodes - 1, rb * 128 // g), min(w.total_nodes - 1, ((rb + 1) * 128 - 1) // g)}
    check_chain_attention(w, nodes=sorted(nodes))


@pytest.mark.parametrize("trees,ctxs", [
    ([W.TreeSpec(2048, [], W.chain_path(1500))], [4096]),
    ([W.TreeSpec(700, [], W.chain_path(699)), W.TreeSpec(2, [], [0]), W.TreeSpec(1300, [], W.chain_path(64))],
     [100, 0, 3000]),
])
def test_chain_lmhead_and_compaction(trees, ctxs):
    """The LM head with anc NULL: argmax as the oracle's, accept length / path /
    bonus as the longest-prefix rule on that argmax (and the planted ones);
    then the in-place compaction (nothing moves) and the buffer compaction,
    bit-exact."""
    E = _E()
    w = W.build("long", seed=53, device="cuda", trees=trees, ctxs=ctxs, **_SMALL)
    x = _placed(w)
    dev = torch.device("cuda")
    i32 = dict(dtype=torch.int32, device=dev)
    ws = E.new_workspace(w.B, w.total_nodes, w.n_q, x["max_ctx"])
    argmax = torch.empty(w.total_nodes, **i32)
    acc = torch.empty(w.B, **i32)
    path = torch.empty((w.B, w.max_T), **i32)
    bonus = torch.empty(w.B, **i32)
    E.ee_lmhead_accept(w.hidden_states, w.lm_w, torch.as_tensor(w.draft_tok, **i32), None, None, None,
                       x["node_off"], w.max_T, argmax, acc, path, bonus, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    rng = np.random.default_rng(1)
    nodes = sorted(set(rng.choice(w.total_nodes, 64, replace=False).tolist()) |
                   {int(w.node_off[s]) + k for s in range(w.B) for k in (0, int(w.planted_accept[s]))})
    U.check_argmax(w, type("S", (), {"argmax": argmax})(), nodes=nodes)
    ra, rp, rb = O.accept_chain(argmax.cpu().numpy(), w.draft_tok, w.node_off, w.max_T)
    np.testing.assert_array_equal(acc.cpu().numpy(), ra)
    np.testing.assert_array_equal(path.cpu().numpy(), rp)
    np.testing.assert_array_equal(bonus.cpu().numpy(), rb)
    np.testing.assert_array_equal(ra, w.planted_accept)
    # in place: a chain is already where compaction puts it
    ctx_out = torch.zeros(w.B, **i32)
    dst = torch.full((w.B, w.max_T), 7, **i32)
    E.ee_kv_compact_inplace(x["kc"], x["vc"], x["bt"], x["ctx"], ctx_out, x["node_off"], path, acc,
                            w.total_nodes, dst, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    rk, rv, rdst, rctx = O.kv_compact_inplace(x["kc_np"], x["vc_np"], w.block_table, w.ctx_len, w.node_off, rp, ra)
    np.testing.assert_array_equal(dst.cpu().numpy(), rdst)
    np.testing.assert_array_equal(ctx_out.cpu().numpy(), rctx)
    assert np.array_equal(U.raw16(x["kc"]), rk) and np.array_equal(U.raw16(x["vc"]), rv)
    assert np.array_equal(rk, x["kc_np"])          # nothing moved
    # from separate draft buffers: every accepted entry is copied
    kc0, vc0 = U.raw16(w.k_cache), U.raw16(w.v_cache)
    kc1 = torch.from_numpy(kc0.copy()).view(torch.bfloat16).to(dev)
    vc1 = torch.from_numpy(vc0.copy()).view(torch.bfloat16).to(dev)
    E.ee_kv_compact(w.k_tree, w.v_tree, kc1, vc1, x["bt"], x["ctx"], ctx_out, x["node_off"], path, acc, dst, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    sk, sv, sdst, sctx = O.kv_compact(U.raw16(w.k_tree), U.raw16(w.v_tree), kc0, vc0, w.block_table, w.ctx_len,
                                      w.node_off, rp, ra)
    np.testing.assert_array_equal(dst.cpu().numpy(), sdst)
    np.testing.assert_array_equal(ctx_out.cpu().numpy(), sctx)
    assert np.array_equal(U.raw16(kc1), sk) and np.array_equal(U.raw16(vc1), sv)


def test_chain_step():
    """VerifyStep on linear drafts (chosen from the workload: drafts above 128
    tokens): set-up places the drafts' K/V in the cache; the step's attention,
    acceptance and compaction match the oracle."""
    E = _E()
    from paper_2506_02780_gb300 import step as S
    trees = [W.TreeSpec(700, [], W.chain_path(699)), W.TreeSpec(2, [], [0]), W.TreeSpec(1300, [], W.chain_path(64))]
    w = W.build("long", seed=54, device="cuda", trees=trees, ctxs=[100, 0, 3000], layers=2, vocab=8192,
                hidden=512, n_q=8, n_kv=2)
    st = S.from_workload(w)
    assert st.chain and st.launches_per_step() == 1 + w.layers + 2
    kc0, vc0 = U.raw16(w.k_cache), U.raw16(w.v_cache)
    st.run()
    torch.cuda.synchronize()
    assert E.ee_read_errors(st.ws) == 0
    U.check_match(w, st)
    for l in range(w.layers):
        ref = O.chain_attention(w.q[l], torch.from_numpy(kc0[l]).view(torch.bfloat16),
                                torch.from_numpy(vc0[l]).view(torch.bfloat16), w.block_table, w.ctx_len,
                                w.node_off)
        U.assert_close(st.attn_out[l].cpu().numpy(), ref, f"chain step attention layer {l}")
    ra, rp, rb = O.accept_chain(st.argmax.cpu().numpy(), w.draft_tok, w.node_off, w.max_T)
    np.testing.assert_array_equal(st.accept_len.cpu().numpy(), ra)
    np.testing.assert_array_equal(st.path.cpu().numpy(), rp)
    np.testing.assert_array_equal(ra, w.planted_accept)
    rk, rv, rdst, rctx = O.kv_compact_inplace(kc0, vc0, w.block_table, w.ctx_len, w.node_off, rp, ra)
    np.testing.assert_array_equal(st.dst_slot.cpu().numpy(), rdst)
    np.testing.assert_array_equal(st.ctx_out.cpu().numpy(), rctx)
