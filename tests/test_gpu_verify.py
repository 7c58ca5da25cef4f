"""GPU parity of ee_lmhead_verify -- the verification rules of Sec. V-C
(greedy, direct, top-k) and the entropy-aware rule of Sec. III-B,
Eq. (entropy) -- against the oracle's verify_accept on trees whose draft
tokens are planted at ranks 0-2 of their parents' distributions."""
import numpy as np
import pytest
import torch

import oracle as O
import workloads as W

pytestmark = pytest.mark.gpu

# 20 nodes: a 6-node reuse chain and three generated branches; the planted path
# runs down the chain and into the first branch
TREE = W.TreeSpec(6, [(2, 6), (4, 5), (0, 3)], [0, 1, 2, 6, 7, 8, 9, 10, 11])


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


def _run(w, mode, k, gen=True, verify=True):
    E = _E()
    dev = "cuda"
    i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device=dev)  # noqa: E731
    total = w.total_nodes
    parent, node_off, draft = i32(w.parent), i32(w.node_off), i32(w.draft_tok)
    depth = torch.empty(total, dtype=torch.int32, device=dev)
    anc = torch.empty((total, 2), dtype=torch.int64, device=dev)
    ws = E.new_workspace(w.B, total, w.n_q, 0)
    E.ee_tree_prepare(parent, node_off, depth, anc, ws)
    out = {n: torch.full(sh, -7, dtype=torch.int32, device=dev)
           for n, sh in (("argmax", (total,)), ("acc", (w.B,)), ("path", (w.B, w.max_T)),
                         ("bonus", (w.B,)), ("topk", (total, k)), ("tau", (total,)))}
    h = torch.full((total,), -1.0, dtype=torch.float32, device=dev)
    if verify:
        gm = torch.as_tensor(w.gen_mask, device=dev) if gen else None
        E.ee_lmhead_verify(w.hidden_states, w.lm_w, draft, parent, depth, anc, node_off, w.max_T, mode,
                           k, out["argmax"], out["acc"], out["path"], out["bonus"], ws, gen_mask=gm,
                           topk_ids=out["topk"], top_tau=out["tau"], h_norm=h)
    else:
        E.ee_lmhead_accept(w.hidden_states, w.lm_w, draft, parent, depth, anc, node_off, w.max_T,
                           out["argmax"], out["acc"], out["path"], out["bonus"], ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    r = {n: t.cpu().numpy() for n, t in out.items()}
    r["h"] = h.cpu().numpy()
    return r


def _check(w, r, mode, k, gen=True):
    """Ranked ids exact where the oracle's top k + 1 logits are separated by more
    than twice the fp32 accumulation bound (else the kernel's ids must carry the
    same logits within it); H_norm within 2e-4; top_tau exact unless k * H_norm
    lies within 1e-3 of an integer (there fp32 and fp64 may round apart);
    acceptance equal to the oracle's rule given the kernel's own top_tau."""
    lg, err = O.lm_head_logits(w.hidden_states, w.lm_w)
    total = w.total_nodes
    n_amb = 0
    for a in range(total):
        ref = O.node_ranking(lg[a], k + 1)
        vals = lg[a][ref]
        e = 2.0 * err[a].max()
        if np.all(np.diff(vals) < -e):
            assert list(r["topk"][a]) == list(ref[:k]), f"node {a}"
        else:
            n_amb += 1
            assert len(set(r["topk"][a].tolist())) == k
            np.testing.assert_allclose(lg[a][r["topk"][a]], vals[:k], atol=e, rtol=0)
        assert r["argmax"][a] == r["topk"][a][0]
        if k >= 2:
            t_ref, h_ref, _ = O.entropy_top_tau(lg[a], k)
            assert abs(r["h"][a] - h_ref) < 2e-4, f"node {a}: H_norm {r['h'][a]} vs {h_ref}"
            if mode == "entropy":
                x = k * h_ref
                if abs(x - round(x)) > 1e-3:
                    assert r["tau"][a] == t_ref, f"node {a}"
                else:
                    assert abs(int(r["tau"][a]) - t_ref) <= 1
        want = {"greedy": 1, "topk": k, "direct": 0}.get(mode)
        if want is not None:
            assert r["tau"][a] == want
    acc, path, bonus, _ = O.verify_accept(
        lg, w.draft_tok, w.parent, w.node_off, mode, k=k, gen_mask=w.gen_mask if gen else None,
        max_T=w.max_T, tau_override=r["tau"] if mode == "entropy" else None)
    np.testing.assert_array_equal(r["acc"], acc)
    np.testing.assert_array_equal(r["path"], path)
    np.testing.assert_array_equal(r["bonus"], bonus)
    return n_amb, acc


def _tiny(seed):
    return W.build("tiny", seed=seed, device="cuda", verify_plant=True, trees=[TREE])


@pytest.mark.parametrize("mode,k", [("greedy", 1), ("greedy", 3), ("direct", 3), ("topk", 1),
                                    ("topk", 3), ("topk", 5), ("entropy", 2), ("entropy", 3),
                                    ("entropy", 5), ("entropy", 8)])
def test_verify_modes_tiny(mode, k):
    w = _tiny(41)
    r = _run(w, mode, k)
    _check(w, r, mode, k)


@pytest.mark.parametrize("seed", [42, 43, 44, 45])
def test_verify_entropy_seeds(seed):
    """Several planted trees: the rules disagree on some of them."""
    w = _tiny(seed)
    accs = {}
    for mode, k in (("greedy", 1), ("topk", 3), ("entropy", 3), ("entropy", 5), ("direct", 3)):
        r = _run(w, mode, k)
        accs[(mode, k)] = _check(w, r, mode, k)[1][0]
    assert accs[("greedy", 1)] <= accs[("entropy", 3)] <= accs[("topk", 3)] <= accs[("direct", 3)]


def test_verify_without_gen_mask():
    w = _tiny(46)
    r = _run(w, "entropy", 3, gen=False)
    _check(w, r, "entropy", 3, gen=False)


def test_verify_greedy_matches_lmhead_accept():
    """The greedy rule of the verification kernel and the plain greedy kernel agree bit for bit."""
    w = W.build("tiny", seed=47, device="cuda")
    a = _run(w, "greedy", 1)
    b = _run(w, "greedy", 1, verify=False)
    for n in ("argmax", "acc", "path", "bonus"):
        np.testing.assert_array_equal(a[n], b[n])
    np.testing.assert_array_equal(a["acc"], w.planted_accept)


def test_verify_batched_two_node_tiles():
    """8 sequences, about 500 nodes: two node tiles of the LM head, each merged
    from the partials of its own CTAs."""
    w = W.build("batched", seed=48, device="cuda", verify_plant=True, layers=1, vocab=8192,
                hidden=512)
    assert w.total_nodes > 256
    r = _run(w, "entropy", 5)
    _check(w, r, "entropy", 5)


@pytest.mark.slow
def test_verify_7b_shapes():
    """Full 7b LM head (vocab 152064, hidden 3584), entropy rule with k = 3 and 5."""
    w = W.build("7b", seed=49, device="cuda", verify_plant=True, layers=1)
    for k in (3, 5):
        r = _run(w, "entropy", k)
        _check(w, r, "entropy", k)


@pytest.mark.parametrize("vocab", [30000, 152064 // 8 * 3])
def test_vocab_tiles_drop_the_rows_of_the_next_tile(vocab):
    """Every CTA takes as many vocabulary tiles; a tile of r < 128 rows still
    runs a 128-row MMA whose last 128 - r rows are the next tile's first rows
    and must be dropped.  The best and second-best rows of node 0 are planted
    at first rows of tiles (each also inside the previous tile's MMA): argmax,
    the top-k list (no id twice) and the acceptance agree with the oracle."""
    w = W.build("tiny", seed=71, device="cuda", verify_plant=True, trees=[TREE], vocab=vocab)
    per_group, n_vt0 = 152, (vocab + 127) // 128
    k_tiles = (n_vt0 + per_group - 1) // per_group
    rows = (vocab + k_tiles * per_group - 1) // (k_tiles * per_group)
    assert 64 <= rows < 128, rows                     # the launch uses rows-high tiles
    top, second = 5 * rows, 9 * rows
    h0 = w.hidden_states[0].float()
    w.lm_w[top] = (h0 / h0.norm() * 64.0).to(torch.bfloat16)
    w.lm_w[second] = (h0 / h0.norm() * 48.0).to(torch.bfloat16)
    for mode, k in (("topk", 4), ("entropy", 3)):
        r = _run(w, mode, k)
        assert r["argmax"][0] == top
        assert list(r["topk"][0][:2]) == [top, second]
        for a in range(w.total_nodes):
            assert len(set(r["topk"][a].tolist())) == k, a
        _check(w, r, mode, k)
    g = _run(w, "greedy", 1, verify=False)            # ee_lmhead_accept
    assert g["argmax"][0] == top
    np.testing.assert_array_equal(g["argmax"], _run(w, "greedy", 1)["argmax"])
