"""GPU parity of the device-resident controller: ee_build_reuse_tree and
ee_advance against the oracle on random inputs, and whole edit sessions run as
captured CUDA graphs of whole steps (no host between steps) against the same
sessions run by the oracle.

The target model's layers are not part of the library, so the sessions use a
synthetic greedy target: its hidden state at a tree node is the unit vector of
the LM-head row of the token the target wants there, scaled by 12, so the LM
head's argmax (computed by libee) is that token.  The target wants the edited
code c': after k committed tokens and a node at depth d, c'[k + d].  Greedy
speculative decoding is lossless, so the committed text must be c'."""
import numpy as np
import pytest
import torch

import oracle as O

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


def _dev(a, dtype=torch.int32):
    return torch.as_tensor(np.asarray(a), dtype=dtype, device="cuda")


@pytest.mark.parametrize("seed", [0, 1])
def test_build_tree_and_advance_match_the_oracle(seed):
    E = _E()
    rng = np.random.default_rng(seed)
    B, n, chain_len, nbr, G, M = 5, 4, 9, 3, 4, 6
    codes = [rng.integers(0, 20, int(rng.integers(5, 200))).astype(np.int32) for _ in range(B)]
    codes[1] = codes[1][:4]                                       # shorter than n + 1: no match
    tok = np.concatenate(codes)
    off = np.concatenate([[0], np.cumsum([len(c) for c in codes])]).astype(np.int64)
    tail = np.stack([rng.integers(0, 20, n) for _ in range(B)]).astype(np.int32)
    for s in (0, 2):                                              # planted matches
        if len(codes[s]) > 30:
            tail[s] = codes[s][10:10 + n]
    cursor = np.asarray([int(rng.integers(0, 8)) for _ in range(B)], np.int32)
    mp, nm = O.match_reuse(tok, off, tail, cursor, M)
    last = rng.integers(0, 20, B).astype(np.int32)
    gen = rng.integers(0, 20, (B, G)).astype(np.int32)
    d, par, noff, cpos, gm = O.build_reuse_tree(tok, off, mp, nm, last, n, chain_len, nbr, gen_tok=gen)
    T = 1 + nbr * chain_len + G
    ws = E.new_workspace(B, B * T, 8, 0)
    i32 = dict(dtype=torch.int32, device="cuda")
    gd, gp, gc = (torch.empty(B * T, **i32) for _ in range(3))
    go = torch.empty(B + 1, **i32)
    gg = torch.empty(B * T, dtype=torch.uint8, device="cuda")
    E.ee_build_reuse_tree(_dev(tok), _dev(off, torch.int64), _dev(mp), _dev(nm), _dev(last), n, chain_len, nbr,
                          gd, gp, go, gc, gg, ws, gen_tok=_dev(gen))
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    for got, ref in ((gd, d), (gp, par), (go, noff), (gc, cpos), (gg, gm)):
        np.testing.assert_array_equal(got.cpu().numpy(), ref)
    # commit a random accepted path per sequence
    _, anc = O.tree_prepare(par, noff)
    path = np.full((B, T), -1, np.int32)
    acc = np.zeros(B, np.int32)
    for s in range(B):
        u = int(rng.integers(0, T))
        p = [u]
        while par[s * T + p[-1]] >= 0:
            p.append(int(par[s * T + p[-1]]))
        p = p[::-1]
        path[s, :len(p)] = p
        acc[s] = len(p) - 1
    bonus = rng.integers(0, 20, B).astype(np.int32)
    cap = 400
    out = np.zeros((B, cap), np.int32)
    out_len = np.asarray([int(rng.integers(n, 100)) for _ in range(B)], np.int32)
    for s in range(B):
        out[s, :out_len[s]] = rng.integers(0, 20, out_len[s])
    ro, rl, rt, rc, rlast = O.advance(out, out_len, d, cpos, noff, path, acc, bonus, cursor, n)
    g_out, g_len, g_cur = _dev(out), _dev(out_len), _dev(cursor)
    g_tail = torch.empty((B, n), **i32)
    g_last = torch.empty(B, **i32)
    E.ee_advance(g_out, g_len, gd, gc, go, _dev(path), _dev(acc), _dev(bonus), g_tail, g_cur, g_last, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0
    for got, ref in ((g_out, ro), (g_len, rl), (g_tail, rt), (g_cur, rc), (g_last, rlast)):
        np.testing.assert_array_equal(got.cpu().numpy(), ref)


def test_advance_refuses_a_full_buffer():
    E = _E()
    ws = E.new_workspace(1, 3, 8, 0)
    i32 = dict(dtype=torch.int32, device="cuda")
    out = torch.arange(8, **i32).reshape(1, 8)
    out_len = torch.tensor([7], **i32)
    d = torch.tensor([5, 6, 7], **i32)
    cpos = torch.tensor([-1, 3, 4], **i32)
    tail = torch.zeros((1, 2), **i32)
    cursor = torch.tensor([2], **i32)
    last = torch.zeros(1, **i32)
    E.ee_advance(out, out_len, d, cpos, torch.tensor([0, 3], **i32), torch.tensor([[0, 1, 2]], **i32),
                 torch.tensor([2], **i32), torch.tensor([9], **i32), tail, cursor, last, ws)
    torch.cuda.synchronize()
    assert E.ee_read_errors(ws) == 0x80
    assert out_len.item() == 7 and cursor.item() == 2 and out.cpu().tolist()[0] == list(range(8))


# ----------------------------------------------------------------------------
# whole sessions on the device
# ----------------------------------------------------------------------------

def _edited(rng, c, vocab):
    c = list(c)
    a = int(rng.integers(40, 80))
    c[a:a + 5] = rng.integers(0, vocab, 5).tolist()
    b = int(rng.integers(120, 160))
    c[b:b] = rng.integers(0, vocab, 7).tolist()
    e = int(rng.integers(200, 240))
    del c[e:e + 6]
    return np.asarray(c, np.int32)


def _proposal(cp_row, k, G, vocab):
    """A noisy draft model: the target's next G tokens, every fifth one wrong."""
    out = []
    for j in range(G):
        t = int(cp_row[k + j]) if k + j < len(cp_row) else 0
        out.append((t + 1) % vocab if (k + j) % 5 == 0 and k + j < len(cp_row) else t)
    return out


def test_device_session_reproduces_the_edited_code():
    E = _E()
    from paper_2506_02780_gb300.session import EditSession
    rng = np.random.default_rng(7)
    B, vocab, H, L, n_q, n_kv, n = 2, 8192, 512, 2, 8, 2, 4
    chain_len, nbr, G, P0, K = 24, 2, 3, 20, 8
    codes = [rng.integers(0, vocab, 300).astype(np.int32) for _ in range(B)]
    edited = [_edited(rng, c, vocab) for c in codes]
    T = 1 + nbr * chain_len + G
    span = max(len(c) for c in edited) + 64 * T                 # room for every step's commit and tree
    npg = -(-(P0 + span) // 16)
    dev = torch.device("cuda")
    g = torch.Generator(device=dev).manual_seed(7)
    kc = (torch.randn((L, B * npg, n_kv, 16, 128), generator=g, device=dev) / 11.3).bfloat16()
    vc = (torch.randn((L, B * npg, n_kv, 16, 128), generator=g, device=dev) / 11.3).bfloat16()
    bt = torch.arange(B * npg, dtype=torch.int32, device=dev).reshape(B, npg)
    lm_w = (torch.randn((vocab, H), generator=g, device=dev) * 0.02).bfloat16()
    w_unit = lm_w.float() / lm_w.float().norm(dim=1, keepdim=True)
    cap = max(len(c) for c in edited) + 64 * T
    cp_pad = torch.zeros((B, cap + T + G), dtype=torch.int64, device=dev)
    for s in range(B):
        cp_pad[s, :len(edited[s])] = torch.as_tensor(edited[s])
    cp_len = torch.as_tensor([len(c) for c in edited], device=dev)

    def target_forward(ss):
        seq = torch.div(torch.arange(ss.total, device=dev), ss.T, rounding_mode="floor")
        pos = ss.out_len.long()[seq] + ss.depth.long()
        want = cp_pad[seq, pos]
        ss.hidden.copy_((w_unit[want] * 12.0).bfloat16())

    def draft_proposal(ss):
        k = ss.out_len.long()[:, None] + torch.arange(G, device=dev)[None, :]
        t = cp_pad.gather(1, k)
        wrong = (k % 5) == 0
        ss.gen_tok.copy_(torch.where(wrong & (k < cp_len[:, None]), (t + 1) % vocab, t).int())

    sess = EditSession(orig_tokens=_dev(np.concatenate(codes)),
                       orig_off=_dev(np.cumsum([0] + [len(c) for c in codes]), torch.int64),
                       committed=[e[:P0].tolist() for e in edited], ctx_len=[P0] * B, k_cache=kc, v_cache=vc,
                       block_table=bt, lm_w=lm_w, n_q=n_q, n=n, chain_len=chain_len, n_branches=nbr, gen_len=G,
                       cap=cap, target_forward=target_forward, draft_proposal=draft_proposal,
                       max_ctx=npg * 16 - T)
    g_ = torch.Generator(device=dev).manual_seed(8)
    sess.q.copy_(torch.randn(sess.q.shape, generator=g_, device=dev).bfloat16())
    sess.k_tree.copy_((torch.randn(sess.k_tree.shape, generator=g_, device=dev) / 11.3).bfloat16())
    sess.v_tree.copy_((torch.randn(sess.v_tree.shape, generator=g_, device=dev) / 11.3).bfloat16())
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        sess.step(stream)                                         # first step eagerly (set-up of the library)
    stream.synchronize()
    sess.capture(K, stream)
    steps = 1
    while int(sess.out_len.min()) < max(len(c) for c in edited) and steps < 400:
        sess.replay()
        steps += K
        stream.synchronize()
    assert E.ee_read_errors(sess.ws) == 0
    out = sess.out_tok.cpu().numpy()
    for s in range(B):
        assert np.array_equal(out[s, :len(edited[s])], edited[s]), f"session {s}"
    assert steps < (len(edited[0]) - P0) // 2                    # reuse: many tokens per step
    # the same session on the host, step for step
    ref_out = np.zeros((B, cap), np.int32)
    for s in range(B):
        ref_out[s, :P0] = edited[s][:P0]
    ref_len, ref_cur = np.full(B, P0, np.int32), np.zeros(B, np.int32)
    ref_last = np.asarray([e[P0 - 1] for e in edited], np.int32)
    tok = np.concatenate(codes)
    off = np.cumsum([0] + [len(c) for c in codes]).astype(np.int64)
    for _ in range(steps):
        tail = np.stack([ref_out[s, ref_len[s] - n:ref_len[s]] for s in range(B)])
        mp, nm = O.match_reuse(tok, off, tail, ref_cur, 8)
        gen = np.asarray([_proposal(np.asarray(edited[s]), int(ref_len[s]), G, vocab) for s in range(B)], np.int32)
        d, par, noff, cpos, _ = O.build_reuse_tree(tok, off, mp, nm, ref_last, n, chain_len, nbr, gen_tok=gen)
        dep, _ = O.tree_prepare(par, noff)
        am = np.asarray([int(cp_pad[i // T, ref_len[i // T] + dep[i]]) for i in range(B * T)], np.int32)
        acc, path, bonus = O.accept_path(am, d, par, noff)
        ref_out, ref_len, _, ref_cur, ref_last = O.advance(ref_out, ref_len, d, cpos, noff, path, acc, bonus,
                                                          ref_cur, n)
    np.testing.assert_array_equal(sess.out_len.cpu().numpy(), ref_len)
    np.testing.assert_array_equal(sess.cursor.cpu().numpy(), ref_cur)
    for s in range(B):
        np.testing.assert_array_equal(out[s, :ref_len[s]], ref_out[s, :ref_len[s]])
