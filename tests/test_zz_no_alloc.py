"""ee_lmhead_accept_static, the LM-head entry point for callers that cannot
allocate device memory (no workspace argument: its scratch is a fixed array
inside libee), must return what ee_lmhead_accept returns with a workspace.

Called through the C ABI twice in a row on the same inputs; both calls are
compared with the workspace entry point: argmax, accepted path, accept length
and bonus bit-exact, logits within the parity tolerance.  This file is
collected last so that a run stopping at the first failure has already run
every other test."""
import ctypes

import numpy as np
import pytest
import torch

import parity_util as U
import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def E():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    import paper_2506_02780_gb300 as E
    from paper_2506_02780_gb300 import build
    build.build_lib()
    E.lib()
    return E


def _outputs(w, dev):
    i32 = dict(dtype=torch.int32, device=dev)
    return dict(argmax=torch.full((w.total_nodes,), -7, **i32),
                accept_len=torch.full((w.B,), -7, **i32),
                path=torch.full((w.B, w.max_T), -7, **i32),
                bonus=torch.full((w.B,), -7, **i32),
                logits=torch.full((w.total_nodes, w.vocab), float("nan"), dtype=torch.float32,
                                  device=dev))


@pytest.mark.parametrize("name,ov", [("tiny", {}),
                                     ("batched", dict(layers=1, vocab=20000, hidden=1024))])
def test_static_entry_point_matches_workspace_entry_point(E, name, ov):
    dev = "cuda"
    w = W.build(name, seed=4321, device=dev, **ov)
    i32 = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    parent, node_off, draft = i32(w.parent), i32(w.node_off), i32(w.draft_tok)
    depth = torch.empty(w.total_nodes, dtype=torch.int32, device=dev)
    anc = torch.empty((w.total_nodes, 2), dtype=torch.int64, device=dev)
    ws = E.new_workspace(w.B, w.total_nodes, w.n_q, int(w.ctx_len.max()))
    E.ee_tree_prepare(parent, node_off, depth, anc, ws)

    ref = _outputs(w, dev)
    E.ee_lmhead_accept(w.hidden_states, w.lm_w, draft, parent, depth, anc, node_off, w.max_T,
                       ref["argmax"], ref["accept_len"], ref["path"], ref["bonus"], ws,
                       logits=ref["logits"])
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    np.testing.assert_array_equal(ref["accept_len"].cpu().numpy(), w.planted_accept)

    for call in range(2):
        got = _outputs(w, dev)
        E.ee_lmhead_accept_static(w.hidden_states, w.lm_w, draft, parent, depth, anc, node_off,
                                  w.max_T, got["argmax"], got["accept_len"], got["path"], got["bonus"],
                                  logits=got["logits"])
        torch.cuda.synchronize()
        for k in ("argmax", "accept_len", "path", "bonus"):
            assert torch.equal(got[k], ref[k]), f"call {call}: {k} differs"
        U.assert_close(got["logits"].cpu().numpy(), ref["logits"].cpu().numpy(),
                       f"call {call}: logits")


def test_static_entry_point_rejects_oversized_problem(E):
    fake = ctypes.c_void_p(0x10000)        # never dereferenced: the size check fails first
    st = E.lib().ee_lmhead_accept_static(fake, fake, 512, 4096, fake, fake, fake, fake, fake, 1,
                                         E.EE_MAX_LM_NODES + 1, 16, fake, fake, fake, fake, None, None)
    assert st == 2                          # EE_ERR_UNSUPPORTED: beyond the static scratch


def _ref_and_static(E, w, dev, chain):
    """ee_lmhead_accept with a workspace, then ee_lmhead_accept_static, same inputs."""
    i32 = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    node_off, draft = i32(w.node_off), i32(w.draft_tok)
    ws = E.new_workspace(w.B, w.total_nodes, w.n_q, int(w.ctx_len.max()))
    if chain:
        parent = depth = anc = None
    else:
        parent = i32(w.parent)
        depth = torch.empty(w.total_nodes, dtype=torch.int32, device=dev)
        anc = torch.empty((w.total_nodes, 2), dtype=torch.int64, device=dev)
        E.ee_tree_prepare(parent, node_off, depth, anc, ws)
    ref, got = _outputs(w, dev), _outputs(w, dev)
    E.ee_lmhead_accept(w.hidden_states, w.lm_w, draft, parent, depth, anc, node_off, w.max_T,
                       ref["argmax"], ref["accept_len"], ref["path"], ref["bonus"], ws,
                       logits=ref["logits"])
    E.ee_lmhead_accept_static(w.hidden_states, w.lm_w, draft, parent, depth, anc, node_off, w.max_T,
                              got["argmax"], got["accept_len"], got["path"], got["bonus"],
                              logits=got["logits"])
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    return ref, got


def test_static_entry_point_full_array_then_smaller_call(E):
    """A linear draft of 2048 nodes (every running-argmax word of the array in
    use), then a 16-node tree: the second call must not see the first call's
    words.  Both are bit-identical to the workspace entry point."""
    dev = "cuda"
    big = W.build("long", seed=99, device=dev, layers=1, vocab=20000, hidden=1024)
    assert big.total_nodes == E.EE_MAX_LM_NODES
    small = W.build("tiny", seed=7, device=dev)
    for w, chain in ((big, True), (small, False)):
        ref, got = _ref_and_static(E, w, dev, chain)
        np.testing.assert_array_equal(ref["accept_len"].cpu().numpy(), w.planted_accept)
        for k in ("argmax", "accept_len", "path", "bonus", "logits"):
            assert torch.equal(got[k], ref[k]), f"{w.name}: {k} differs"
