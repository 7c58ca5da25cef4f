"""The seeded input generators produce the configurations as stated (CPU only).

Shapes, tree structure, context and code lengths, value distributions and the
planted structure (matches, accept lengths, repeated segments) of every
configuration, at one layer and without the LM-head weight where the full
configuration is large.
"""
import numpy as np
import pytest
import torch

import workloads as W


def _chain_and_branches(w, s):
    o, T = int(w.node_off[s]), int(w.node_off[s + 1] - w.node_off[s])
    par = [int(x) for x in w.parent[o:o + T]]
    chain = 1
    while chain < T and par[chain] == chain - 1:
        chain += 1
    branches, i = [], chain
    while i < T:
        attach, j = par[i], i + 1
        while j < T and par[j] == j - 1:
            j += 1
        branches.append((attach, j - i))
        i = j
    return T, chain, branches


def test_tiny():
    w = W.build("tiny")
    assert (w.B, w.n_q, w.n_kv, w.head_dim, w.hidden, w.vocab, w.layers, w.n) == (1, 8, 2, 128, 512, 4096, 1, 4)
    c = w.seq_tokens(0)
    assert len(c) == 400 and c.min() >= 0 and c.max() < 4096
    assert int(w.ctx_len[0]) == 512
    assert _chain_and_branches(w, 0) == (16, 12, [(0, 4)])
    # prefix = c[0:300] with edits; the tail is its last 4 tokens, planted at p = 296
    assert list(w.tail[0]) == list(c[296:300]) and int(w.planted_match[0]) == 296
    # K/V ~ N(0,1)/sqrt(128), W ~ N(0, 0.02^2)
    assert abs(w.k_cache.float().std().item() - 128 ** -0.5) < 0.01
    assert abs(w.lm_w.float().std().item() - 0.02) < 0.002
    assert w.k_cache.dtype == torch.bfloat16 and w.lm_w.dtype == torch.bfloat16


def test_7b_shapes():
    w = W.build("7b", layers=1, lm_head=False)
    assert (w.n_q, w.n_kv, w.hidden, w.vocab, W.SHAPES["7b"]["layers"]) == (28, 4, 3584, 152064, 28)
    assert len(w.seq_tokens(0)) == 3000 and int(w.ctx_len[0]) == 4096
    assert _chain_and_branches(w, 0) == (64, 48, [(0, 8), (24, 8)])
    assert int(w.planted_accept[0]) == 30
    assert w.k_cache.shape[2:] == (4, W.PAGE, 128)


def test_batched_ragged():
    w = W.build("batched", layers=1, lm_head=False)
    assert w.B == 8 and (w.n_q, w.n_kv, w.hidden, w.vocab) == (28, 4, 3584, 152064)
    ctx = w.ctx_len.astype(int)
    assert ctx.min() >= 1024 and ctx.max() <= 16384 and len(set(ctx.tolist())) == 8
    for s in range(w.B):
        T, chain, branches = _chain_and_branches(w, s)
        assert 32 <= T <= 96
        assert 0.5 - 1.0 / T <= chain / T <= 0.9 + 1.0 / T
        assert 1 <= len(branches) <= 2 and sum(b[1] for b in branches) == T - chain
        assert len(w.seq_tokens(s)) == int(round(0.8 * ctx[s]))


def test_33b_long_file():
    w = W.build("33b", layers=1, lm_head=False)
    assert (w.n_q, w.n_kv, w.hidden, w.vocab, W.SHAPES["33b"]["layers"]) == (56, 8, 7168, 32256, 62)
    assert int(w.ctx_len[0]) == 32768 and len(w.seq_tokens(0)) == 28000
    T, chain, branches = _chain_and_branches(w, 0)
    assert (T, chain) == (128, 112) and len(branches) == 4 and all(b[1] == 4 for b in branches)


def test_long_reuse_draft():
    w = W.build("long", layers=1, lm_head=False)
    assert int(w.ctx_len[0]) == 4096 and len(w.seq_tokens(0)) == 8000
    assert _chain_and_branches(w, 0) == (2048, 2048, [])
    assert int(w.planted_accept[0]) == 1500


@pytest.mark.parametrize("n", [2, 4, 8])
def test_sweep(n):
    w = W.build("sweep", layers=1, n=n)
    assert w.B == 32 and w.n == n and w.tail.shape == (32, n)
    assert all(len(w.seq_tokens(s)) == 65536 for s in range(w.B))
    assert w.orig_tokens.min() >= 0 and w.orig_tokens.max() < 152064
    acc = w.planted_accept.astype(int)
    assert acc.min() >= 0 and acc.max() <= 127          # accepted-path lengths acc + 1 in [1, 128]
    assert all(_chain_and_branches(w, s) == (128, 128, []) for s in range(w.B))
    real = int((w.planted_match >= 0).sum())
    assert 24 <= real <= 32                              # about 90% of tails come from the code
    for s in np.nonzero(w.planted_match >= 0)[0]:
        p = int(w.planted_match[s])
        assert list(w.tail[s]) == list(w.seq_tokens(s)[p:p + n])


def test_sweep_repeated_segments():
    """30% of each code lies in copies of earlier 8-token spans that no copy
    overwrites: at least 30% of positions lie in an 8-gram that occurs earlier
    (the configuration's "30% of n-grams repeated"), and every recorded copy is
    an exact repeat of its source."""
    w = W.build("sweep", layers=1, B=3)
    for s in range(w.B):
        c = w.seq_tokens(s)
        seen, rep = set(), np.zeros(len(c), bool)
        for p in range(len(c) - 7):
            key = c[p:p + 8].tobytes()
            if key in seen:
                rep[p:p + 8] = True
            seen.add(key)
        assert 0.30 <= rep.mean() <= 0.34, rep.mean()
