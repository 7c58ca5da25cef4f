"""fp64 CPU oracle for the EfficientEdit verification step -- TEST INFRASTRUCTURE.

This package is the plain, slow, obviously-correct statement of what one
verification step of edit-oriented speculative decoding computes (EfficientEdit,
arXiv 2506.02780, Sec. III-A "Reuse" and Eq. (piecewise)).  It exists to check
the CUDA library against; it is not part of the product path.  Only the test
suite, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference
leg may import it.  It shares no code with the CUDA path and imports nothing
from the product package.

Every floating-point step runs in fp64 on exact fp64 copies of the bf16 inputs.
Library primitives (numpy matmul, argmax) serve as single steps; nothing is
blocked, fused or reordered beyond what each definition states.

Parity status per function (what pins it, from outside this file, in
tests/test_oracle_pins.py):
  match_reuse      pinned: brute-force byte search, planted matches, closed forms
  tree_prepare     pinned: walk-up brute force, chain/star closed forms
  tree_attention   pinned: torch SDPA in fp64 over each node's linear path,
                   single-key and equal-key closed forms, page-order invariance
  lm_head_argmax   pinned: planted argmax targets, duplicated-row ties,
                   pure-Python dot products on a tiny case; the fp32
                   accumulation bound against four fp32 summation orders and
                   hand-built near ties (the candidate sets)
  accept_path      pinned: token-by-token replay of Eq. (piecewise), brute force
                   over all root-to-node paths, hand-worked golden cases
  kv_compact       pinned: sequential append into a slot dictionary, canaries
  tree_kv_to_cache / tree_kv_from_cache
                   pinned: round trip, slot-dictionary placement
  chain_attention  pinned: equals tree_attention on chain trees (T <= 128) with the
                   draft placed in the cache; torch SDPA (fp64, causal) over
                   prefix + draft for longer drafts
  accept_chain     pinned: equals accept_path on chain parents; token replay
  build_reuse_tree / advance
                   pinned: hand-worked trees and commits; a whole edit session
                   (match, tree, a synthetic greedy target, acceptance, commit)
                   reproduces the target's own greedy text (lossless greedy
                   speculative decoding) from several starting points
  kv_compact_inplace
                   pinned: equals kv_compact on the committed positions after
                   tree_kv_to_cache (random trees and paths), chains move
                   nothing, a hand-worked overlapping move
  entropy_top_tau  pinned: closed forms of Eq. (entropy) / top_tau (H=0, uniform)
  verify_accept    pinned: reduces to accept_path (greedy; top-1; all-reuse trees),
                   top-V = direct, brute force over root-to-node paths, H = 0 and
                   uniform top-k distributions
"""
from .ee_oracle import (  # noqa: F401
    PAGE,
    match_reuse,
    tree_prepare,
    anc_to_sets,
    tree_attention,
    lm_head_logits,
    lm_head_argmax,
    accept_path,
    kv_compact,
    tree_kv_to_cache,
    tree_kv_from_cache,
    kv_compact_inplace,
    chain_attention,
    accept_chain,
    build_reuse_tree,
    advance,
    entropy_top_tau,
    VERIFY_MODES,
    node_ranking,
    verify_accept,
    verify_step,
)
