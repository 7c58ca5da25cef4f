"""Why the attention keeps P to about 2^-17 and writes fp32 (CPU only).

The tolerance on attention outputs is max abs 2e-2 and mean relative error
sum|g - r| / sum|r| <= 1e-3 against fp64.  On 7B-shaped rows (a 4096-key
context plus a 64-node draft, queries N(0,1), keys and values N(0,1)/sqrt(128),
all bf16, seven query heads per KV head) this test measures, in numpy/torch
against an fp64 reference, the error of each rounding the kernel could make:

  P rounded to bf16 before P.V       ~1.5e-3  (breaks 1e-3 alone)
  the output rounded to bf16          ~1.4e-3  (breaks 1e-3 alone)
  P rounded to fp16 (V too)           ~1.9e-4
  P as a bf16 head + bf16 tail        ~2e-6    (what the kernel does, V as stored)

so the kernel splits P into two bf16 parts for the tensor cores and writes fp32.
"""
import torch


def _rows():
    g = torch.Generator().manual_seed(0)
    ctx, T, g_heads, d = 4096, 64, 7, 128
    k = (torch.randn(ctx + T, d, generator=g) / d ** 0.5).to(torch.bfloat16).double()
    v = (torch.randn(ctx + T, d, generator=g) / d ** 0.5).to(torch.bfloat16).double()
    q = torch.randn(T * g_heads, d, generator=g).to(torch.bfloat16).double()
    s = (q @ k.T) / d ** 0.5
    p = torch.exp(s - s.max(dim=1, keepdim=True).values)
    l = p.sum(1, keepdim=True)
    return p, l, v, (p @ v) / l


def _mean_rel(x, ref):
    return ((x - ref).abs().sum() / ref.abs().sum()).item()


def test_single_bf16_roundings_break_the_tolerance_and_the_split_does_not():
    p, l, v, ref = _rows()
    p_bf16 = p.float().to(torch.bfloat16).double()
    e_p_bf16 = _mean_rel((p_bf16 @ v) / l, ref)
    e_out_bf16 = _mean_rel(ref.float().to(torch.bfloat16).double(), ref)
    e_p_fp16 = _mean_rel((p.float().half().double() @ v.float().half().double()) / l, ref)
    head = p.float().to(torch.bfloat16).float()
    tail = (p.float() - head).to(torch.bfloat16).double()
    e_split = _mean_rel(((head.double() + tail) @ v) / l, ref)
    assert e_p_bf16 > 1e-3 and e_out_bf16 > 1e-3
    assert e_p_fp16 < 5e-4
    assert e_split < 1e-5
    # the split carries P to about 2^-17 relative
    rel = ((head.double() + tail) - p.float().double()).abs() / p.float().double().clamp_min(1e-30)
    assert rel.max().item() <= 2.0 ** -16
