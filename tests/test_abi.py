"""The C-ABI library builds, loads and exports every entry point include/ee.h
declares; host-side argument checks reject bad calls before any launch
(CPU only: nothing here touches a GPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    import paper_2506_02780_gb300 as E
    from paper_2506_02780_gb300 import build
    if not os.path.exists(E.LIB_PATH):
        try:
            build.build_lib()
        except RuntimeError as e:   # no nvcc on this machine
            pytest.skip(str(e))
    return E.lib()


def declared_symbols():
    with open(os.path.join(ROOT, "include", "ee.h")) as f:
        text = f.read()
    return sorted(set(re.findall(r"^\s*(?:ee_status|size_t|const char\*)\s+(ee_\w+)\(", text, re.M)))


def test_header_declares_the_boundary():
    syms = declared_symbols()
    for name in ("ee_match_reuse", "ee_tree_prepare", "ee_tree_verify_attn", "ee_lmhead_accept",
                 "ee_kv_compact", "ee_workspace_size", "ee_workspace_init", "ee_read_errors",
                 "ee_version", "ee_status_string"):
        assert name in syms


def test_every_declared_symbol_is_exported(L):
    for name in declared_symbols():
        assert hasattr(L, name), name
    import paper_2506_02780_gb300 as E
    assert set(E.EXPORTS) <= set(declared_symbols())


def test_version_and_status_strings(L):
    assert b"sm_103a" in L.ee_version()
    assert L.ee_status_string(0) == b"ok"
    assert L.ee_status_string(5) == b"workspace too small"


def test_workspace_size(L):
    """A fixed head (error word, LM-head ticket, running argmax words: 8 bytes
    per node up to EE_MAX_LM_NODES), the LM-head verification partials (152
    CTAs x 256 nodes x 80-byte records (8 top-k values, 8 ids, max and sum,
    padded to 16 bytes), then one 8-byte
    pruning threshold per node, the finalize step's 8 ranked ids and top_tau
    per node), 1 MiB for the split reuse-span match (tickets and per-CTA
    records), and, when the
    context is split, one attention partial slot per CTA: 128 rows x 128 fp32
    + 128 x (m, l) + a 256-byte counter trailer, for at most B x n_q row blocks
    x 16 chunks, and at least two per SM (152) for the balanced launch.
    Independent of the node count."""
    head = L.ee_workspace_size(1, 64, 28, 128, 0)
    assert head == L.ee_workspace_size(8, 2048, 56, 128, 0)
    assert head % 256 == 0
    assert head == 16896 + 152 * 256 * 80 + 8 * 2048 + 4 * 2048 * 8 + 4 * 2048 + (1 << 20)
    slot = 128 * 128 * 4 + 128 * 8 + 256
    assert slot % 256 == 0
    for B, n_q, ctx in ((1, 28, 4096), (8, 56, 262144), (3, 8, 16), (1, 8, 512)):
        n_slots = max(B * n_q * 16, 2 * 152)
        assert L.ee_workspace_size(B, 64, n_q, 128, ctx) == head + n_slots * slot
        assert L.ee_workspace_size(B, 2048, n_q, 128, ctx) == head + n_slots * slot
    assert L.ee_workspace_size(-1, 64, 28, 128, 16) == 0
    assert L.ee_workspace_size(1, 64, 28, 128, -1) == 0


FAKE = ctypes.c_void_p(0x10000)   # never dereferenced: every call below fails validation first


def test_lmhead_verify_rejects_bad_mode_or_k(L):
    f = L.ee_lmhead_verify
    def call(mode, k):
        return f(FAKE, FAKE, 64, 100, FAKE, FAKE, FAKE, FAKE, FAKE, None, 1, 4, 4, mode, k,
                 FAKE, None, None, None, FAKE, FAKE, FAKE, None, FAKE, 1 << 30, None)
    assert call(4, 3) == 1 and call(-1, 3) == 1          # no such mode
    assert call(2, 0) == 1 and call(2, 9) == 1           # k out of 1..8
    assert call(3, 1) == 1                               # entropy needs k >= 2 (ln k > 0)


def test_attn_plan_rejects_bad_args(L):
    out = [ctypes.c_int32(0) for _ in range(4)]
    ptrs = [ctypes.byref(x) for x in out]
    f = L.ee_attn_plan
    for inplace in (0, 1):
        assert f(0, 64, 28, 4, 4096, inplace, *ptrs) == 1          # no sequence
        assert f(1, 129, 28, 4, 4096, inplace, *ptrs) == 1         # tree larger than 128 nodes
        assert f(1, 64, 28, 5, 4096, inplace, *ptrs) == 1          # n_q not a multiple of n_kv
        assert f(1, 64, 28, 4, -1, inplace, *ptrs) == 1            # negative context
        assert f(1, 64, 28, 4, 4096, inplace, None, *ptrs[1:]) == 1
    assert f(1, 64, 28, 4, 4096, 3, *ptrs) == 1                    # inplace is 0, 1 or 2 (chain)
    assert f(1, 2049, 28, 4, 4096, 2, *ptrs) == 1                  # a chain above EE_MAX_CHAIN
    assert f(1, 129, 28, 4, 4096, 1, *ptrs) == 1                   # a tree above EE_MAX_TREE


def test_inplace_entry_points_reject_bad_args(L):
    ws = ctypes.c_void_p(0x20000)
    a = L.ee_tree_verify_attn_inplace
    base = [FAKE, FAKE, FAKE, 10, FAKE, 4, FAKE, 40, FAKE, FAKE, 1, 16, 16, 8, 2, 128,
            ctypes.c_float(0.088), FAKE, ws, 1 << 26, None]
    assert a(*base[:7], 49, *base[8:]) == 1          # max_ctx + max_T = 65 > max_pages * 16
    bad = list(base); bad[15] = 64
    assert a(*bad) == 2                               # head_dim other than 128
    bad = list(base); bad[0] = None
    assert a(*bad) == 1
    c = L.ee_kv_compact_inplace
    cb = [FAKE, FAKE, 10 * 2 * 16 * 128, 2, 10, FAKE, 4, FAKE, ctypes.c_void_p(0x30000), FAKE, FAKE, FAKE,
          1, 16, 16, 2, 128, FAKE, ws, 1 << 26, None]
    bad = list(cb); bad[8] = FAKE
    assert c(*bad) == 1                               # ctx_len_out aliases ctx_len_in
    bad = list(cb); bad[14] = 2049
    assert c(*bad) == 1                               # a path above EE_MAX_CHAIN
    bad = list(cb); bad[16] = 64
    assert c(*bad) == 2
    bad = list(cb); bad[19] = 64
    assert c(*bad) == 5                               # workspace below the head


def test_match_rejects_bad_args(L):
    f = L.ee_match_reuse
    # n = 0, n too large, max_matches = 0
    assert f(FAKE, FAKE, 1, FAKE, 0, FAKE, 4, FAKE, FAKE, FAKE, 1 << 20, None) == 1
    assert f(FAKE, FAKE, 1, FAKE, 33, FAKE, 4, FAKE, FAKE, FAKE, 1 << 20, None) == 1
    assert f(FAKE, FAKE, 1, FAKE, 4, FAKE, 0, FAKE, FAKE, FAKE, 1 << 20, None) == 1
    assert f(FAKE, None, 1, FAKE, 4, FAKE, 4, FAKE, FAKE, FAKE, 1 << 20, None) == 1
    assert f(FAKE, FAKE, 1, FAKE, 4, FAKE, 4, FAKE, FAKE, FAKE, 64, None) == 5      # workspace
    assert f(None, None, 0, None, 4, None, 4, None, None, None, 0, None) == 0      # B = 0: no-op


def test_attention_rejects_bad_args(L):
    f = L.ee_tree_verify_attn
    ws = 1 << 30
    args = [FAKE] * 5 + [10, FAKE, 4, FAKE, 64, FAKE, FAKE, 1, 16, 16, 8, 2, 128,
                         ctypes.c_float(0.088), FAKE, FAKE, ws, None]
    bad_hd = list(args); bad_hd[17] = 64
    assert f(*bad_hd) == 2                                   # head_dim must be 128
    bad_g = list(args); bad_g[15] = 7                        # n_q not a multiple of n_kv
    assert f(*bad_g) == 2
    bad_T = list(args); bad_T[14] = 129
    assert f(*bad_T) == 2
    bad_ctx = list(args); bad_ctx[9] = 65                    # max_ctx > max_pages * 16
    assert f(*bad_ctx) == 1
    bad_scale = list(args); bad_scale[18] = ctypes.c_float(0.0)
    assert f(*bad_scale) == 1
    unaligned = list(args); unaligned[0] = ctypes.c_void_p(0x10002)
    assert f(*unaligned) == 1
    small = list(args); small[21] = 1024
    assert f(*small) == 5


def test_lmhead_rejects_bad_args(L):
    f = L.ee_lmhead_accept
    base = [FAKE, FAKE, 3584, 152064] + [FAKE] * 5 + [1, 64, 64] + [FAKE] * 4 + [None, FAKE, 1 << 20, None]
    h7 = list(base); h7[2] = 3583
    assert f(*h7) == 2                                       # hidden not a multiple of 8
    many = list(base); many[10] = 4096
    assert f(*many) == 2                                     # too many nodes for one call
    nul = list(base); nul[4] = None
    assert f(*nul) == 1


def test_compact_rejects_aliasing_ctx(L):
    f = L.ee_kv_compact
    args = [FAKE, FAKE, 1024, FAKE, FAKE, 8192, 2, 10, FAKE, 4, FAKE, ctypes.c_void_p(0x20000), FAKE,
            FAKE, FAKE, 1, 16, 4, 128, FAKE, FAKE, 1 << 20, None]
    alias = list(args); alias[11] = args[10]
    assert f(*alias) == 1
    hd = list(args); hd[18] = 96
    assert f(*hd) == 2


def test_selftest_timeout_rejects_bad_args(L):
    f = L.ee_selftest_timeout
    assert f(None, 1 << 20, FAKE, None) == 1                     # no workspace
    assert f(FAKE, 1 << 20, None, None) == 1                     # no output
    assert f(FAKE, 64, FAKE, None) == 1                          # below the fixed head
    assert f(ctypes.c_void_p(0x10008), 1 << 20, FAKE, None) == 1   # ws not 256-aligned
    assert f(FAKE, 1 << 20, ctypes.c_void_p(0x10004), None) == 1   # out not 8-aligned


def test_chain_entry_points_reject_bad_args(L):
    ws = ctypes.c_void_p(0x20000)
    a = L.ee_chain_verify_attn
    base = [FAKE, FAKE, FAKE, 200, FAKE, 160, FAKE, 512, FAKE, 1, 2048, 2048, 8, 2, 128,
            ctypes.c_float(0.088), FAKE, ws, 1 << 26, None]
    bad = list(base); bad[11] = 2049
    assert a(*bad) == 2                               # draft above EE_MAX_CHAIN
    bad = list(base); bad[5] = 159
    assert a(*bad) == 1                               # 512 + 2048 positions need 160 pages
    bad = list(base); bad[14] = 64
    assert a(*bad) == 2
    # the LM head takes linear drafts with anc NULL (parent / depth may be NULL too)
    f = L.ee_lmhead_accept
    lm = [FAKE, FAKE, 512, 4096, FAKE, None, None, None, FAKE, 1, 2048, 2049] + [FAKE] * 4 + [None, ws, 1 << 26, None]
    assert f(*lm) == 2                                # max_T above EE_MAX_CHAIN
    tree = [FAKE, FAKE, 512, 4096, FAKE, None, FAKE, FAKE, FAKE, 1, 2048, 129] + [FAKE] * 4 + [None, ws, 1 << 26, None]
    assert f(*tree) == 2                              # a tree above EE_MAX_TREE
    v = L.ee_lmhead_verify
    assert v(FAKE, FAKE, 512, 4096, FAKE, None, None, None, FAKE, None, 1, 64, 64, 0, 1,
             FAKE, None, None, None, FAKE, FAKE, FAKE, None, ws, 1 << 26, None) == 1   # rules need a tree


def test_controller_rejects_bad_args(L):
    ws = ctypes.c_void_p(0x20000)
    b = L.ee_build_reuse_tree
    base = [FAKE, FAKE, 2, FAKE, FAKE, 4, FAKE, 4, 24, 4, None, 0] + [FAKE] * 5 + [ws, 1 << 26, None]
    bad = list(base); bad[8] = 32
    assert b(*bad) == 2                                # 1 + 4 x 32 nodes > 128
    bad = list(base); bad[11] = 3
    assert b(*bad) == 1                                # a generated branch without tokens
    bad = list(base); bad[7] = 33
    assert b(*bad) == 1                                # n above EE_MAX_NGRAM
    bad = list(base); bad[18] = 64
    assert b(*bad) == 5
    a = L.ee_advance
    abase = [FAKE, FAKE, 4096, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 2, 194, 97, 4, FAKE, FAKE, FAKE, ws, 1 << 26, None]
    bad = list(abase); bad[11] = 129
    assert a(*bad) == 1                                # a tree above EE_MAX_TREE
    bad = list(abase); bad[2] = 0
    assert a(*bad) == 1
    bad = list(abase); bad[13] = None
    assert a(*bad) == 1


def test_lmhead_packing_sizes_and_checks(L):
    """The tile-ordered weights take ceil(V / 128) * 128 rows of ceil(H / 64) * 64
    columns; bad sizes, pointers and short buffers are rejected before a launch."""
    assert L.ee_lmhead_packed_bytes(152064, 3584) == 152064 * 3584 * 2
    assert L.ee_lmhead_packed_bytes(1000, 512) == 1024 * 512 * 2
    assert L.ee_lmhead_packed_bytes(1000, 520) == 1024 * 576 * 2
    assert L.ee_lmhead_packed_bytes(1000, 12) == 0 and L.ee_lmhead_packed_bytes(0, 512) == 0
    f = L.ee_lmhead_pack_weights
    n = L.ee_lmhead_packed_bytes(1000, 512)
    assert f(None, 1000, 512, FAKE, n, None) == 1
    assert f(FAKE, 1000, 512, None, n, None) == 1
    assert f(FAKE, 1000, 512, FAKE, n - 16, None) == 1            # buffer too small
    assert f(ctypes.c_void_p(0x10002), 1000, 512, FAKE, n, None) == 1
    assert f(FAKE, 1000, 12, FAKE, n, None) == 2                  # hidden not a multiple of 8
    assert f(FAKE, 0, 512, FAKE, n, None) == 1
    g = L.ee_lmhead_accept_packed
    base = [FAKE, FAKE, 3584, 152064] + [FAKE] * 5 + [1, 64, 64] + [FAKE] * 4 + [None, FAKE, 1 << 20, None]
    h7 = list(base); h7[2] = 3583
    assert g(*h7) == 2                                            # as ee_lmhead_accept
    small = list(base); small[18] = 64
    assert g(*small) == 5
