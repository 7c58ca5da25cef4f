"""Python binding of libee, the sm_103a library for one EfficientEdit
verification step (arXiv 2506.02780, Sec. III-A).

Every function here has the name of the C entry point it wraps (include/ee.h)
and only marshals arguments: torch CUDA tensors become raw device pointers,
the current torch stream becomes the launch stream, and a non-zero status
becomes an ``EEError``.  All computation runs in the library's kernels; there
is no CPU or PyTorch fallback, and importing fails loudly when libee.so is
missing.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libee.so")

EE_PAGE = 16
EE_HEAD_DIM = 128
EE_MAX_TREE = 128
EE_MAX_LM_NODES = 2048

STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported configuration", 3: "CUDA error",
          4: "device error word set", 5: "workspace too small"}
DEVERR = {0x01: "MATCH_ARGS", 0x02: "TREE", 0x04: "PAGE", 0x08: "CTX", 0x10: "FP16_RANGE",
          0x20: "TIMEOUT", 0x40: "PATH", 0x80: "OVERFLOW"}
DEVERR_TIMEOUT = 0x20

EXPORTS = ("ee_version", "ee_status_string", "ee_workspace_size", "ee_workspace_init",
           "ee_read_errors", "ee_match_reuse", "ee_tree_prepare", "ee_tree_verify_attn", "ee_attn_plan",
           "ee_lmhead_accept", "ee_lmhead_verify", "ee_lmhead_accept_static", "ee_kv_compact",
           "ee_selftest_timeout", "ee_tree_verify_attn_inplace", "ee_kv_compact_inplace",
           "ee_chain_verify_attn", "ee_build_reuse_tree", "ee_advance", "ee_lmhead_packed_bytes",
           "ee_lmhead_pack_weights", "ee_lmhead_accept_packed")

VERIFY_MODES = {"greedy": 0, "direct": 1, "topk": 2, "entropy": 3}


class EEError(RuntimeError):
    def __init__(self, fn, status, bits=0):
        msg = f"{fn}: {STATUS.get(status, status)}"
        if bits:
            msg += " [" + ",".join(v for k, v in DEVERR.items() if bits & k) + "]"
        super().__init__(msg)
        self.status = status
        self.bits = bits


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int32
_I64 = ctypes.c_int64
_SZ = ctypes.c_size_t
_F = ctypes.c_float

_SIGS = {
    "ee_version": ([], ctypes.c_char_p),
    "ee_status_string": ([_I], ctypes.c_char_p),
    "ee_workspace_size": ([_I, _I, _I, _I, _I], _SZ),
    "ee_workspace_init": ([_P, _SZ, _P], _I),
    "ee_read_errors": ([_P, _P, ctypes.POINTER(_I)], _I),
    "ee_match_reuse": ([_P, _P, _I, _P, _I, _P, _I, _P, _P, _P, _SZ, _P], _I),
    "ee_tree_prepare": ([_P, _P, _I, _I, _P, _P, _P, _SZ, _P], _I),
    "ee_tree_verify_attn": ([_P, _P, _P, _P, _P, _I, _P, _I, _P, _I, _P, _P, _I, _I, _I, _I, _I, _I,
                             _F, _P, _P, _SZ, _P], _I),
    "ee_attn_plan": ([_I, _I, _I, _I, _I, _I, ctypes.POINTER(_I), ctypes.POINTER(_I), ctypes.POINTER(_I),
                      ctypes.POINTER(_I)], _I),
    "ee_tree_verify_attn_inplace": ([_P, _P, _P, _I, _P, _I, _P, _I, _P, _P, _I, _I, _I, _I, _I, _I, _F, _P,
                                     _P, _SZ, _P], _I),
    "ee_chain_verify_attn": ([_P, _P, _P, _I, _P, _I, _P, _I, _P, _I, _I, _I, _I, _I, _I, _F, _P, _P, _SZ, _P],
                             _I),
    "ee_build_reuse_tree": ([_P, _P, _I, _P, _P, _I, _P, _I, _I, _I, _P, _I, _P, _P, _P, _P, _P, _P, _SZ, _P],
                            _I),
    "ee_advance": ([_P, _P, _I, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _P, _P, _P, _P, _SZ, _P], _I),
    "ee_kv_compact_inplace": ([_P, _P, _I64, _I, _I, _P, _I, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P,
                               _SZ, _P], _I),
    "ee_lmhead_accept": ([_P, _P, _I, _I, _P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _P, _P, _SZ,
                          _P], _I),
    "ee_lmhead_verify": ([_P, _P, _I, _I, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P, _P, _P, _P,
                          _P, _P, _P, _P, _SZ, _P], _I),
    "ee_lmhead_accept_static": ([_P, _P, _I, _I, _P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _P,
                                 _P], _I),
    "ee_lmhead_packed_bytes": ([_I, _I], _SZ),
    "ee_lmhead_pack_weights": ([_P, _I, _I, _P, _SZ, _P], _I),
    "ee_lmhead_accept_packed": ([_P, _P, _I, _I, _P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _P, _P, _SZ,
                                 _P], _I),
    "ee_kv_compact": ([_P, _P, _I64, _P, _P, _I64, _I, _I, _P, _I, _P, _P, _P, _P, _P, _I, _I, _I, _I,
                       _P, _P, _SZ, _P], _I),
    "ee_selftest_timeout": ([_P, _SZ, _P, _P], _I),
}


def lib():
    """The loaded libee.so (ctypes CDLL).  Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2506_02780_gb300.build` (needs nvcc)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGS.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _p(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libee takes CUDA tensors only")
    if not t.is_contiguous():
        raise ValueError("libee takes contiguous tensors only")
    return ctypes.c_void_p(t.data_ptr())


def _check(t, dtype, name):
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _ok(fn, status):
    if status != 0:
        raise EEError(fn, status)


def ee_version() -> str:
    return lib().ee_version().decode()


def ee_workspace_size(B, total_nodes, n_q, head_dim, max_ctx) -> int:
    return int(lib().ee_workspace_size(B, total_nodes, n_q, head_dim, max_ctx))


def ee_workspace_init(ws, stream=None):
    _ok("ee_workspace_init", lib().ee_workspace_init(_p(ws), ws.numel(), _stream(stream)))


def ee_read_errors(ws, stream=None) -> int:
    """Synchronise, return and clear the device error word (0 = no error)."""
    bits = _I(0)
    st = lib().ee_read_errors(_p(ws), _stream(stream), ctypes.byref(bits))
    if st not in (0, 4):
        raise EEError("ee_read_errors", st)
    return int(bits.value)


def ee_selftest_timeout(ws, out, stream=None):
    """Run the bounded-wait self-test; `out` is a device int64[7] (see ee.h)."""
    _check(out, torch.int64, "out")
    if out.numel() < 7:
        raise ValueError("out needs 7 int64")
    _ok("ee_selftest_timeout", lib().ee_selftest_timeout(_p(ws), ws.numel(), _p(out), _stream(stream)))


def new_workspace(B, total_nodes, n_q, max_ctx, device="cuda", stream=None):
    """Allocate (through torch) and zero a workspace big enough for these sizes."""
    n = ee_workspace_size(B, total_nodes, n_q, EE_HEAD_DIM, max_ctx)
    ws = torch.empty(n, dtype=torch.uint8, device=device)
    ee_workspace_init(ws, stream)
    return ws


def ee_match_reuse(orig_tokens, orig_off, tail, cursor, max_matches, match_pos, n_matches, ws,
                   stream=None):
    _check(orig_tokens, torch.int32, "orig_tokens")
    _check(orig_off, torch.int64, "orig_off")
    B, n = tail.shape
    st = lib().ee_match_reuse(_p(orig_tokens), _p(orig_off), B, _p(tail), n, _p(cursor), max_matches,
                              _p(match_pos), _p(n_matches), _p(ws), ws.numel(), _stream(stream))
    _ok("ee_match_reuse", st)


def ee_tree_prepare(parent, node_off, depth, anc, ws, stream=None):
    _check(parent, torch.int32, "parent")
    _check(anc, torch.int64, "anc (uint64 bits stored as int64)")
    B = node_off.numel() - 1
    st = lib().ee_tree_prepare(_p(parent), _p(node_off), B, parent.numel(), _p(depth), _p(anc), _p(ws),
                               ws.numel(), _stream(stream))
    _ok("ee_tree_prepare", st)


def ee_tree_verify_attn(q, k_tree, v_tree, k_cache, v_cache, block_table, ctx_len, max_ctx, node_off,
                        anc, max_T, scale, out, ws, stream=None):
    for t, nm in ((q, "q"), (k_tree, "k_tree"), (v_tree, "v_tree"), (k_cache, "k_cache"),
                  (v_cache, "v_cache")):
        _check(t, torch.bfloat16, nm)
    _check(out, torch.float32, "out")
    total, n_q, d = q.shape
    n_kv = k_tree.shape[1]
    num_pages = k_cache.shape[0]
    B, max_pages = block_table.shape
    st = lib().ee_tree_verify_attn(_p(q), _p(k_tree), _p(v_tree), _p(k_cache), _p(v_cache), num_pages,
                                   _p(block_table), max_pages, _p(ctx_len), max_ctx, _p(node_off),
                                   _p(anc), B, total, max_T, n_q, n_kv, d, float(scale), _p(out),
                                   _p(ws), ws.numel(), _stream(stream))
    _ok("ee_tree_verify_attn", st)


def ee_tree_verify_attn_inplace(q, k_cache, v_cache, block_table, ctx_len, max_ctx, node_off, anc, max_T,
                                scale, out, ws, stream=None):
    """Tree attention with the tree's K/V at cache positions ctx + i (one layer)."""
    for t, nm in ((q, "q"), (k_cache, "k_cache"), (v_cache, "v_cache")):
        _check(t, torch.bfloat16, nm)
    _check(out, torch.float32, "out")
    total, n_q, d = q.shape
    num_pages, n_kv = k_cache.shape[0], k_cache.shape[1]
    B, max_pages = block_table.shape
    st = lib().ee_tree_verify_attn_inplace(_p(q), _p(k_cache), _p(v_cache), num_pages, _p(block_table),
                                           max_pages, _p(ctx_len), max_ctx, _p(node_off), _p(anc), B, total,
                                           max_T, n_q, n_kv, d, float(scale), _p(out), _p(ws), ws.numel(),
                                           _stream(stream))
    _ok("ee_tree_verify_attn_inplace", st)


def ee_chain_verify_attn(q, k_cache, v_cache, block_table, ctx_len, max_ctx, node_off, max_T, scale, out, ws,
                         stream=None):
    """Causal attention of linear drafts (up to EE_MAX_CHAIN tokens) whose K/V sit
    at cache positions ctx + i (one layer)."""
    for t, nm in ((q, "q"), (k_cache, "k_cache"), (v_cache, "v_cache")):
        _check(t, torch.bfloat16, nm)
    _check(out, torch.float32, "out")
    total, n_q, d = q.shape
    num_pages, n_kv = k_cache.shape[0], k_cache.shape[1]
    B, max_pages = block_table.shape
    st = lib().ee_chain_verify_attn(_p(q), _p(k_cache), _p(v_cache), num_pages, _p(block_table), max_pages,
                                    _p(ctx_len), max_ctx, _p(node_off), B, total, max_T, n_q, n_kv, d,
                                    float(scale), _p(out), _p(ws), ws.numel(), _stream(stream))
    _ok("ee_chain_verify_attn", st)


def ee_attn_plan(B, max_T, n_q, n_kv, max_ctx, inplace=False) -> dict:
    """The launch plan ee_tree_verify_attn (inplace False / 0),
    ee_tree_verify_attn_inplace (True / 1) or ee_chain_verify_attn ("chain" / 2)
    uses for these sizes."""
    kv = 2 if inplace == "chain" else int(inplace)
    v = [_I(0) for _ in range(4)]
    st = lib().ee_attn_plan(B, max_T, n_q, n_kv, max_ctx, kv, *[ctypes.byref(x) for x in v])
    _ok("ee_attn_plan", st)
    return {"splits": v[0].value, "chunk": v[1].value,
            "mode": ("single", "cluster", "cooperative", "balanced")[v[2].value], "ctas": v[3].value}


def ee_lmhead_accept(hidden, lm_w, draft_tok, parent, depth, anc, node_off, max_T, argmax, accept_len,
                     path, bonus, ws, logits=None, stream=None):
    _check(hidden, torch.bfloat16, "hidden")
    _check(lm_w, torch.bfloat16, "lm_w")
    total, H = hidden.shape
    V = lm_w.shape[0]
    B = node_off.numel() - 1
    st = lib().ee_lmhead_accept(_p(hidden), _p(lm_w), H, V, _p(draft_tok), _p(parent), _p(depth),
                                _p(anc), _p(node_off), B, total, max_T, _p(argmax), _p(accept_len),
                                _p(path), _p(bonus), _p(logits), _p(ws), ws.numel(), _stream(stream))
    _ok("ee_lmhead_accept", st)


def ee_lmhead_packed_bytes(vocab, hidden_dim):
    """Bytes of the tile-ordered LM-head weights for these sizes (0: not supported)."""
    return int(lib().ee_lmhead_packed_bytes(int(vocab), int(hidden_dim)))


def ee_lmhead_pack_weights(lm_w, packed, stream=None):
    """Write `lm_w` ([vocab][hidden] bf16) into `packed` (a bf16 tensor of at least
    ee_lmhead_packed_bytes(vocab, hidden) bytes) in the LM head's tile order."""
    _check(lm_w, torch.bfloat16, "lm_w")
    _check(packed, torch.bfloat16, "packed")
    V, H = lm_w.shape
    st = lib().ee_lmhead_pack_weights(_p(lm_w), V, H, _p(packed), packed.numel() * 2, _stream(stream))
    _ok("ee_lmhead_pack_weights", st)


def ee_lmhead_accept_packed(hidden, lm_w_packed, vocab, draft_tok, parent, depth, anc, node_off, max_T, argmax,
                            accept_len, path, bonus, ws, logits=None, stream=None):
    """ee_lmhead_accept with the weights packed by ee_lmhead_pack_weights (the
    vocabulary size is an argument: the packed array is padded)."""
    _check(hidden, torch.bfloat16, "hidden")
    _check(lm_w_packed, torch.bfloat16, "lm_w_packed")
    total, H = hidden.shape
    B = node_off.numel() - 1
    st = lib().ee_lmhead_accept_packed(_p(hidden), _p(lm_w_packed), H, int(vocab), _p(draft_tok), _p(parent),
                                       _p(depth), _p(anc), _p(node_off), B, total, max_T, _p(argmax),
                                       _p(accept_len), _p(path), _p(bonus), _p(logits), _p(ws), ws.numel(),
                                       _stream(stream))
    _ok("ee_lmhead_accept_packed", st)


def ee_lmhead_verify(hidden, lm_w, draft_tok, parent, depth, anc, node_off, max_T, mode, k, argmax,
                     accept_len, path, bonus, ws, gen_mask=None, topk_ids=None, top_tau=None,
                     h_norm=None, logits=None, stream=None):
    """LM head + argmax + acceptance under a verification rule: ``mode`` is one of
    "greedy", "direct", "topk", "entropy" (or its EE_VERIFY_* number);
    ``gen_mask`` uint8 marks edit content (None: every node)."""
    _check(hidden, torch.bfloat16, "hidden")
    _check(lm_w, torch.bfloat16, "lm_w")
    if gen_mask is not None:
        _check(gen_mask, torch.uint8, "gen_mask")
    total, H = hidden.shape
    V = lm_w.shape[0]
    B = node_off.numel() - 1
    m = VERIFY_MODES[mode] if isinstance(mode, str) else int(mode)
    st = lib().ee_lmhead_verify(_p(hidden), _p(lm_w), H, V, _p(draft_tok), _p(parent), _p(depth),
                                _p(anc), _p(node_off), _p(gen_mask), B, total, max_T, m, k,
                                _p(argmax), _p(topk_ids), _p(top_tau), _p(h_norm), _p(accept_len),
                                _p(path), _p(bonus), _p(logits), _p(ws), ws.numel(), _stream(stream))
    _ok("ee_lmhead_verify", st)


def ee_lmhead_accept_static(hidden, lm_w, draft_tok, parent, depth, anc, node_off, max_T, argmax,
                            accept_len, path, bonus, logits=None, stream=None):
    """ee_lmhead_accept without a workspace, for callers that cannot allocate
    device memory: the scratch is a fixed 16,640-byte array inside libee shared
    by every call (calls must not overlap on the GPU)."""
    _check(hidden, torch.bfloat16, "hidden")
    _check(lm_w, torch.bfloat16, "lm_w")
    total, H = hidden.shape
    V = lm_w.shape[0]
    B = node_off.numel() - 1
    st = lib().ee_lmhead_accept_static(_p(hidden), _p(lm_w), H, V, _p(draft_tok), _p(parent),
                                       _p(depth), _p(anc), _p(node_off), B, total, max_T, _p(argmax),
                                       _p(accept_len), _p(path), _p(bonus), _p(logits),
                                       _stream(stream))
    _ok("ee_lmhead_accept_static", st)


def ee_kv_compact(k_tree, v_tree, k_cache, v_cache, block_table, ctx_len_in, ctx_len_out, node_off,
                  path, accept_len, dst_slot, ws, stream=None):
    """k_tree/v_tree [L, total, n_kv, d]; k_cache/v_cache [L, num_pages, n_kv, PAGE, d]."""
    L, total, n_kv, d = k_tree.shape
    num_pages = k_cache.shape[1]
    B, max_pages = block_table.shape
    max_T = path.shape[1]
    st = lib().ee_kv_compact(_p(k_tree), _p(v_tree), total * n_kv * d, _p(k_cache), _p(v_cache),
                             num_pages * n_kv * EE_PAGE * d, L, num_pages, _p(block_table), max_pages,
                             _p(ctx_len_in), _p(ctx_len_out), _p(node_off), _p(path), _p(accept_len),
                             B, max_T, n_kv, d, _p(dst_slot), _p(ws), ws.numel(), _stream(stream))
    _ok("ee_kv_compact", st)


def ee_kv_compact_inplace(k_cache, v_cache, block_table, ctx_len_in, ctx_len_out, node_off, path,
                          accept_len, total_nodes, dst_slot, ws, stream=None):
    """k_cache/v_cache [L, num_pages, n_kv, PAGE, d] holding the tree's K/V at ctx + i."""
    L, num_pages, n_kv, _, d = k_cache.shape
    B, max_pages = block_table.shape
    max_T = path.shape[1]
    st = lib().ee_kv_compact_inplace(_p(k_cache), _p(v_cache), num_pages * n_kv * EE_PAGE * d, L, num_pages,
                                     _p(block_table), max_pages, _p(ctx_len_in), _p(ctx_len_out),
                                     _p(node_off), _p(path), _p(accept_len), B, int(total_nodes), max_T, n_kv,
                                     d, _p(dst_slot), _p(ws), ws.numel(), _stream(stream))
    _ok("ee_kv_compact_inplace", st)


def ee_build_reuse_tree(orig_tokens, orig_off, match_pos, n_matches, last_tok, n, chain_len, n_branches,
                        draft_tok, parent, node_off, cpos, gen_mask, ws, gen_tok=None, stream=None):
    """Next draft tree: root, one reuse chain per match point, a generated branch."""
    B = orig_off.numel() - 1
    gen_len = 0 if gen_tok is None else gen_tok.shape[1]
    _ok("ee_build_reuse_tree",
        lib().ee_build_reuse_tree(_p(orig_tokens), _p(orig_off), B, _p(match_pos), _p(n_matches),
                                  match_pos.shape[1], _p(last_tok), n, chain_len, n_branches, _p(gen_tok), gen_len,
                                  _p(draft_tok), _p(parent), _p(node_off), _p(cpos), _p(gen_mask), _p(ws),
                                  ws.numel(), _stream(stream)))


def ee_advance(out_tok, out_len, draft_tok, cpos, node_off, path, accept_len, bonus, tail, cursor, last_tok, ws,
               stream=None):
    """Commit a step: accepted tokens + bonus appended, tail / cursor / root updated."""
    B, cap = out_tok.shape
    _ok("ee_advance",
        lib().ee_advance(_p(out_tok), _p(out_len), cap, _p(draft_tok), _p(cpos), _p(node_off), _p(path),
                         _p(accept_len), _p(bonus), B, draft_tok.numel(), path.shape[1], tail.shape[1], _p(tail),
                         _p(cursor), _p(last_tok), _p(ws), ws.numel(), _stream(stream)))
