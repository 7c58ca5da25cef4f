"""Planted mistakes in the fp64 oracle are caught by its pins (CPU only).

Each mutant below copies the oracle module, rewrites one function with a
plausible slip -- a dropped term, an off-by-one, a wrong index or operand, a
reversed tie rule -- and runs the pins of tests/test_oracle_pins.py against the
copy.  The test passes when at least one of the named pins fails on the mutant,
so every pin set demonstrably constrains the arithmetic it claims to.  A
control run rebuilds each rewritten function from its unchanged source by the
same mechanism and checks that the same pins all pass, so a broken rewrite
cannot make every mutant look caught.

The mistakes are planted on the CPU, in a throw-away copy of the oracle; the
oracle on disk and the CUDA library are never touched.
"""
import inspect
import itertools
import textwrap
import types

import pytest

import oracle.ee_oracle as ORIG
import test_oracle_pins as PINS


def _expand(fn):
    """Every argument set of a (possibly parametrized) pin function."""
    axes = []
    for mark in getattr(fn, "pytestmark", []):
        if mark.name != "parametrize":
            continue
        names, values = mark.args[0], mark.args[1]
        names = [s.strip() for s in names.split(",")] if isinstance(names, str) else list(names)
        rows = [v if len(names) > 1 else (v,) for v in values]
        axes.append([dict(zip(names, r)) for r in rows])
    for combo in itertools.product(*axes):
        kw = {}
        for part in combo:
            kw.update(part)
        yield kw


def _module_with(func_name, old=None, new=None):
    """A fresh copy of the oracle module with ``func_name`` re-made from its
    source, after replacing every ``old`` by ``new`` (unchanged when old is None)."""
    mod = types.ModuleType("oracle_mutant")
    mod.__dict__.update({k: v for k, v in vars(ORIG).items() if not k.startswith("__")})
    src = textwrap.dedent(inspect.getsource(getattr(ORIG, func_name)))
    if old is not None:
        assert src.count(old) >= 1, f"{func_name}: the text to mutate is no longer in the oracle: {old!r}"
        src = src.replace(old, new)
    exec(compile(src, f"<mutant {func_name}>", "exec"), mod.__dict__)
    # functions copied from the original still see the original module's globals;
    # re-bind them to the copy so that a call chain reaches the rewritten function
    for k, v in list(mod.__dict__.items()):
        if isinstance(v, types.FunctionType) and v.__module__ == ORIG.__name__:
            mod.__dict__[k] = types.FunctionType(v.__code__, mod.__dict__, v.__name__, v.__defaults__,
                                                 v.__closure__)
    return mod


def _failing_pins(mod, pins, monkeypatch):
    """Names of the pins (with arguments) that fail when the oracle is ``mod``."""
    monkeypatch.setattr(PINS, "O", mod)
    failed = []
    for name in pins:
        fn = getattr(PINS, name)
        for kw in _expand(fn):
            try:
                fn(**kw)
            except Exception as e:  # an assertion, or a crash the slip causes
                failed.append(f"{name}{kw if kw else ''}: {type(e).__name__}")
                break
    return failed


ATTN_PINS = ["test_attention_each_node_is_causal_attention_over_its_path",
             "test_attention_chain_equals_masked_sdpa", "test_attention_single_key_returns_value",
             "test_attention_equal_keys_average_values", "test_attention_page_order_invariance",
             "test_attention_gqa_head_map"]
LM_PINS = ["test_lm_head_pure_python_dot", "test_lm_head_planted_argmax",
           "test_lm_head_duplicate_rows_lowest_id", "test_lm_head_identity_closed_form",
           "test_lm_head_fp32_accumulation_stays_within_the_bound",
           "test_lm_head_candidates_hold_every_argmax_within_the_bound",
           "test_lm_head_candidates_at_a_gap_between_one_and_two_bounds"]
ACCEPT_PINS = ["test_accept_golden", "test_accept_chain_replay_random", "test_accept_tree_bruteforce_random",
               "test_accept_planted"]
COMPACT_PINS = ["test_compact_golden", "test_compact_sequential_append_and_canary"]
MATCH_PINS = ["test_match_golden", "test_match_bruteforce_sweep", "test_match_closed_form_constant_code",
              "test_match_planted_tiny"]
TREE_PINS = ["test_tree_prepare_closed_forms", "test_tree_prepare_walk_up"]
VERIFY_PINS = ["test_entropy_golden", "test_verify_greedy_is_accept_path",
               "test_verify_top1_is_greedy_and_reuse_only_is_greedy", "test_verify_top_vocab_is_direct",
               "test_verify_bruteforce_random", "test_verify_entropy_closed_forms"]
INPLACE_PINS = ["test_tree_kv_placement_round_trip", "test_compact_inplace_equals_append",
                "test_compact_inplace_chain_moves_nothing", "test_compact_inplace_overlapping_moves_golden"]
CHAIN_PINS = ["test_chain_attention_equals_tree_attention_on_chains",
              "test_chain_attention_long_draft_is_causal_sdpa", "test_accept_chain_equals_tree_rule_on_chains"]
SESSION_PINS = ["test_build_reuse_tree_golden", "test_advance_golden", "test_session_reproduces_the_target_text"]

# (id, function, text, replacement, pins expected to catch it)
MUTANTS = [
    # match (Sec. III-A prefix matching)
    ("match_no_trailing_draft_token", "match_reuse", "pos + n < len(c)", "pos + n <= len(c)", MATCH_PINS),
    ("match_skips_cursor_position", "match_reuse", "pos >= cursor[s]", "pos > cursor[s]", MATCH_PINS),
    ("match_one_token_short", "match_reuse", "windows == tail[s][None, :]",
     "windows[:, :-1] == tail[s][None, :-1]", MATCH_PINS),
    # tree structure
    ("tree_node_not_its_own_ancestor", "tree_prepare", "sets.append(sets[p] | {i})",
     "sets.append(set(sets[p]))", TREE_PINS),
    ("tree_depth_not_incremented", "tree_prepare", "depth[o + i] = depth[o + p] + 1",
     "depth[o + i] = depth[o + p]", TREE_PINS),
    # tree attention
    ("attention_scale_dropped", "tree_attention", "scale = 1.0 / math.sqrt(d)", "scale = 1.0", ATTN_PINS),
    ("attention_scale_squared", "tree_attention", "scale = 1.0 / math.sqrt(d)", "scale = 1.0 / d", ATTN_PINS),
    ("attention_gqa_head_map_modulo", "tree_attention", "h // g == hk", "h % n_kv == hk", ATTN_PINS),
    ("attention_keys_as_values", "tree_attention", "out[o + i, h] = p @ vals", "out[o + i, h] = p @ keys",
     ATTN_PINS),
    ("attention_node_misses_own_key", "tree_attention", "path = sorted(anc_to_sets(anc[o + i]))",
     "path = sorted(anc_to_sets(anc[o + i]) - {i}) or [i]", ATTN_PINS),
    ("attention_context_one_short", "_context_kv", "[:ctx]", "[:ctx - 1]", ATTN_PINS),
    ("attention_softmax_unnormalised", "tree_attention", "p /= p.sum()", "p /= 1.0", ATTN_PINS),
    # LM head and decode()
    ("argmax_ties_to_highest_id", "lm_head_argmax", "am = np.argmax(logits, axis=1)",
     "am = logits.shape[1] - 1 - np.argmax(logits[:, ::-1], axis=1)", LM_PINS),
    ("lm_head_vocab_reversed", "lm_head_logits", "logits = x @ w.T", "logits = (w @ x.T).T[:, ::-1]",
     LM_PINS),
    ("lm_head_bound_too_tight", "lm_head_logits", "err = 2.0 * x.shape[1] * _U32", "err = 1e-3 * _U32",
     LM_PINS),
    ("candidates_ignore_own_error", "lm_head_argmax", "logits[i] + err[i] >= lo", "logits[i] >= lo", LM_PINS),
    # acceptance, Eq. (piecewise)
    ("accept_judged_at_child", "accept_path", "int(argmax[o + p])", "int(argmax[o + i])", ACCEPT_PINS),
    ("accept_bonus_from_draft", "accept_path", "bonus[s] = int(argmax[o + best])",
     "bonus[s] = int(draft_tok[o + best])", ACCEPT_PINS),
    ("accept_ignores_rejected_parent", "accept_path", "accepted[i] = accepted[p] and",
     "accepted[i] =", ACCEPT_PINS),
    ("accept_equal_depth_to_highest_id", "accept_path", "depth[i] > depth[best]",
     "depth[i] >= depth[best]", ACCEPT_PINS),
    # compaction
    ("compact_slot_off_by_one", "kv_compact", "pos = ctx + k", "pos = ctx + k + 1", COMPACT_PINS),
    ("compact_copies_kth_node", "kv_compact", "src = int(node_off[s]) + node", "src = int(node_off[s]) + k",
     COMPACT_PINS),
    ("compact_context_misses_root", "kv_compact", "ctx_out[s] = ctx + int(accept_len[s]) + 1",
     "ctx_out[s] = ctx + int(accept_len[s])", COMPACT_PINS),
    # entropy-aware verification, Eq. (entropy) and top_tau
    ("entropy_floor_for_ceil", "entropy_top_tau", "math.ceil(k * h)", "math.floor(k * h)", VERIFY_PINS),
    ("entropy_not_normalised", "entropy_top_tau", "/ math.log(k))", ")", VERIFY_PINS),
    ("verify_reuse_judged_by_mode", "verify_accept", "if not gen[o + i]:", "if False:", VERIFY_PINS),
    ("verify_topk_one_short", "verify_accept", "tau[a] = kk\n", "tau[a] = kk - 1\n", VERIFY_PINS),
    # in-place K/V
    ("inplace_placement_by_depth", "tree_kv_to_cache", "_slot(block_table, s, ctx + i,",
     "_slot(block_table, s, ctx + max(i - 1, 0),", INPLACE_PINS),
    ("inplace_moves_in_reverse", "kv_compact_inplace", "for k in range(int(accept_len[s]) + 1):",
     "for k in reversed(range(int(accept_len[s]) + 1)):", INPLACE_PINS),
    # long reuse drafts
    ("chain_causal_mask_excludes_self", "chain_attention", "ctx + i + 1]", "ctx + i]", CHAIN_PINS),
    ("chain_accept_judged_one_late", "accept_chain", "int(argmax[o + j])", "int(argmax[o + j + 1])",
     CHAIN_PINS),
    # Reuse <-> Generate controller
    ("controller_chain_starts_at_match", "build_reuse_tree", "q = int(match_pos[s, b]) + n + j",
     "q = int(match_pos[s, b]) + n - 1 + j", SESSION_PINS),
    ("controller_cursor_not_past_q", "advance", "cursor[s] = q + 1", "cursor[s] = q", SESSION_PINS),
    ("controller_branch_without_match", "build_reuse_tree", "has = b < min(int(n_matches[s]), match_pos.shape[1])",
     "has = b < match_pos.shape[1]", SESSION_PINS),
    ("controller_branch_from_absent_match", "build_reuse_tree",
     "has = b < min(int(n_matches[s]), match_pos.shape[1])",
     "has = b < min(int(n_matches[s]), match_pos.shape[1]) or b == 0", SESSION_PINS),
    ("controller_root_position_without_match", "build_reuse_tree", "if n_matches[s] > 0:", "if True:",
     SESSION_PINS),
    ("controller_root_position_past_match", "build_reuse_tree", "cpos[o] = match_pos[s, 0] + n - 1",
     "cpos[o] = match_pos[s, 0] + n", SESSION_PINS),
    ("advance_recommits_root", "advance", "for k in range(1, a + 1)", "for k in range(0, a + 1)", SESSION_PINS),
    ("advance_tail_before_bonus", "advance", "tail[s] = out[s, out_len[s] - n:out_len[s]]",
     "tail[s] = out[s, out_len[s] - n - 1:out_len[s] - 1]", SESSION_PINS),
    ("inplace_reads_values_as_keys", "tree_kv_from_cache", "kt[:, o + i] = kc[:L, page, :, off, :]",
     "kt[:, o + i] = vc[:L, page, :, off, :]", INPLACE_PINS),
]


@pytest.mark.parametrize("func", sorted({m[1] for m in MUTANTS}))
def test_unmutated_copy_passes_its_pins(func, monkeypatch):
    pins = sorted({p for m in MUTANTS if m[1] == func for p in m[4]})
    failed = _failing_pins(_module_with(func), pins, monkeypatch)
    assert not failed, f"the copy of {func} fails its pins without a mutation: {failed}"


@pytest.mark.parametrize("mid,func,old,new,pins", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_is_caught(mid, func, old, new, pins, monkeypatch):
    failed = _failing_pins(_module_with(func, old, new), pins, monkeypatch)
    assert failed, f"mutant {mid} ({func}: {old!r} -> {new!r}) passes every pin in {pins}"
