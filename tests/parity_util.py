"""Comparison helpers for the GPU parity tests: run the CUDA step through the
C ABI and check it against the fp64 oracle on the same seeded inputs.

Tolerances (written here, used by every parity test):
  - integer outputs (match positions/counts, depth, ancestor masks, accepted
    path, accept length, bonus, compaction slots, compacted cache bytes):
    bit-exact;
  - argmax: equal to the oracle's wherever the fp64 top-2 gap exceeds the fp32
    accumulation bound, otherwise one of the tied candidates;
  - attention outputs and logits: max abs error <= 2e-2 and mean relative
    error sum|g - r| / sum|r| <= 1e-3 (bf16 inputs, fp32 accumulation).
"""
import numpy as np
import torch

import oracle as O

ATOL = 2e-2
MEAN_REL = 1e-3


def close_stats(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    m = ~np.isnan(ref)
    d = np.abs(got[m] - ref[m])
    return float(d.max()) if d.size else 0.0, float(d.sum() / max(np.abs(ref[m]).sum(), 1e-300))


def assert_close(got, ref, what):
    mx, mr = close_stats(got, ref)
    assert mx <= ATOL and mr <= MEAN_REL, f"{what}: max abs {mx:.3e}, mean rel {mr:.3e}"
    return mx, mr


def raw16(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy()


def check_match(w, step):
    pos, cnt = O.match_reuse(w.orig_tokens, w.orig_off, w.tail, w.cursor, w.max_matches)
    np.testing.assert_array_equal(step.match_pos.cpu().numpy(), pos)
    np.testing.assert_array_equal(step.n_matches.cpu().numpy(), cnt)


def check_tree(w, step):
    depth, anc = O.tree_prepare(w.parent, w.node_off)
    np.testing.assert_array_equal(step.depth.cpu().numpy(), depth)
    np.testing.assert_array_equal(step.anc.cpu().numpy().view(np.uint64), anc)
    return anc


def check_attention(w, step, layers, anc, nodes=None):
    stats = []
    for l in layers:
        ref = O.tree_attention(w.q[l], w.k_tree[l], w.v_tree[l], w.k_cache[l], w.v_cache[l],
                               w.block_table, w.ctx_len, w.node_off, anc, nodes=nodes)
        got = step.attn_out[l].cpu().numpy()
        stats.append(assert_close(got, ref, f"attention layer {l}"))
    return stats


def check_argmax(w, step, nodes=None, logits=None):
    """argmax valid per the oracle (exact where unique); logits within tolerance."""
    hid = w.hidden_states if nodes is None else w.hidden_states[torch.as_tensor(nodes)]
    am_ref, cands, lg = O.lm_head_argmax(hid, w.lm_w)
    got = step.argmax.cpu().numpy()
    sel = np.arange(w.total_nodes) if nodes is None else np.asarray(nodes)
    n_amb = 0
    for k, i in enumerate(sel):
        if len(cands[k]) == 1:
            assert got[i] == am_ref[k], f"node {i}: argmax {got[i]} != {am_ref[k]}"
        else:
            n_amb += 1
            assert got[i] in set(cands[k].tolist()), f"node {i}: {got[i]} not a near-tie candidate"
    if logits is not None:
        assert_close(logits.cpu().numpy()[sel], lg, "logits")
    return n_amb


def check_accept(w, step):
    """Acceptance of the GPU argmax equals the oracle's walk on the same argmax;
    planted accept lengths are reproduced."""
    am = step.argmax.cpu().numpy()
    acc, path, bonus = O.accept_path(am, w.draft_tok, w.parent, w.node_off, w.max_T)
    np.testing.assert_array_equal(step.accept_len.cpu().numpy(), acc)
    np.testing.assert_array_equal(step.path.cpu().numpy(), path)
    np.testing.assert_array_equal(step.bonus.cpu().numpy(), bonus)
    return acc, path


def check_compact(w, step, k_cache0, v_cache0, acc, path):
    L = w.layers
    kc, vc, dst, ctx_out = O.kv_compact(raw16(w.k_tree), raw16(w.v_tree), k_cache0, v_cache0,
                                        w.block_table, w.ctx_len, w.node_off, path, acc)
    np.testing.assert_array_equal(step.dst_slot.cpu().numpy(), dst)
    np.testing.assert_array_equal(step.ctx_out.cpu().numpy(), ctx_out)
    for l in range(L):
        assert np.array_equal(raw16(w.k_cache[l]), kc[l]), f"k_cache layer {l}"
        assert np.array_equal(raw16(w.v_cache[l]), vc[l]), f"v_cache layer {l}"
