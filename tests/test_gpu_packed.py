"""GPU: the tile-ordered LM-head weights (ee_lmhead_pack_weights) hold W's
blocks exactly where the header says, and the LM head reading them
(ee_lmhead_accept_packed) returns bit-identical argmax, acceptance and logits
to ee_lmhead_accept on row-major W -- same products, same summation order."""
import numpy as np
import pytest
import torch

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


@pytest.mark.parametrize("V,H", [(1000, 520), (128, 64), (4096, 512)])
def test_packed_layout(V, H):
    E = _E()
    g = torch.Generator(device="cuda").manual_seed(V + H)
    w = torch.randn(V, H, generator=g, device="cuda").to(torch.bfloat16)
    n = E.ee_lmhead_packed_bytes(V, H)
    assert n == -(-V // 128) * 128 * -(-H // 64) * 64 * 2
    packed = torch.full((n // 2,), float("nan"), dtype=torch.bfloat16, device="cuda")
    E.ee_lmhead_pack_weights(w, packed)
    torch.cuda.synchronize()
    wv = w.view(torch.int16).cpu().numpy()
    nvt, nkb = -(-V // 128), -(-H // 64)
    full = np.zeros((nvt * 128, nkb * 64), dtype=np.int16)
    full[:V, :H] = wv
    want = full.reshape(nvt, 128, nkb, 64).transpose(0, 2, 1, 3).reshape(-1)
    np.testing.assert_array_equal(packed.view(torch.int16).cpu().numpy(), want)


def _lm(w, packed):
    """argmax, acceptance and logits of one LM-head call on workload w."""
    E = _E()
    from paper_2506_02780_gb300 import step as S
    st = S.from_workload(w, packed_lm=False)
    st.run(layers=[])    # the tree's depth and ancestor masks (no attention); the LM heads below are compared
    x = st.inp
    total, V = w.total_nodes, w.vocab
    lg = torch.empty((total, V), dtype=torch.float32, device="cuda")
    out = [torch.full(sh, -7, dtype=torch.int32, device="cuda")
           for sh in ((total,), (w.B,), (w.B, w.max_T), (w.B,))]
    chain = st.chain
    tree = (None, None, None) if chain else (x["parent"], st.depth, st.anc)
    if packed:
        pk = torch.empty(E.ee_lmhead_packed_bytes(V, w.hidden) // 2, dtype=torch.bfloat16, device="cuda")
        E.ee_lmhead_pack_weights(x["lm_w"], pk)
        E.ee_lmhead_accept_packed(x["hidden"], pk, V, x["draft_tok"], *tree, x["node_off"], w.max_T, *out, st.ws,
                                  logits=lg)
    else:
        E.ee_lmhead_accept(x["hidden"], x["lm_w"], x["draft_tok"], *tree, x["node_off"], w.max_T, *out, st.ws,
                           logits=lg)
    torch.cuda.synchronize()
    assert E.ee_read_errors(st.ws) == 0
    return [t.cpu() for t in out] + [lg.cpu()]


@pytest.mark.parametrize("name,ov", [
    ("tiny", {}),
    ("tiny", {"vocab": 1000}),                        # vocabulary not a multiple of 128
    ("7b", {"layers": 1}),
    ("long", {"layers": 1, "vocab": 20000, "hidden": 1024}),   # a 2048-token chain: anc NULL
])
def test_packed_lm_head_bit_identical(name, ov):
    w = W.build(name, seed=81, device="cuda", **ov)
    a, b = _lm(w, False), _lm(w, True)
    for x, y in zip(a, b):
        assert torch.equal(x, y)
