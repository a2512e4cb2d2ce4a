"""GPU parity of groups of more than 8 query heads per value head (the multi-query and
grouped-query layouts of Section 3: every head of a group reads the same cached value rows).

The tensor-core decodes serve such a group with sibling CTAs of up to 8 heads each (the bf16
decode puts 4 heads on each of their eight compute warps); every floating-point output is
checked against the fp64 oracle at |gpu - oracle| <= 2e-3 + 1e-2 |oracle|, the appended rows
bit-exact. The CUDA-core kernel serves groups of up to 8 heads and must reject larger ones
without launching.
"""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300.workloads import bf16_bits
from tests import _gpu
from tests._gpu import assert_parity, decode, oracle_decode, shape_of, to_dev
from tests._inputs import tiny

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


SHAPES = [
    dict(B=2, Hq=32, Hkv=1, D=128, P=16, lens=(3000, 17)),        # MQA, 32 query heads
    dict(B=2, Hq=128, Hkv=8, D=128, P=32, lens=(1000, 257)),      # GQA 16 (128 / 8)
    dict(B=3, Hq=24, Hkv=2, D=128, P=16, lens=(0, 700, 129)),     # group 12: blocks of 8 and 4
    dict(B=1, Hq=64, Hkv=2, D=128, P=64, lens=(2222,)),           # group 32, P 64
    dict(B=2, Hq=48, Hkv=2, D=128, P=32, lens=(1500, 64)),        # group 24: three blocks of 8
    dict(B=3, Hq=20, Hkv=1, D=128, P=16, lens=(900, 0, 3000)),    # group 20: 8, 8 and 4, MQA
]


@pytest.mark.parametrize("si", range(len(SHAPES)))
@pytest.mark.parametrize("splits", [1, 3, 0])
def test_large_group_decode_matches_oracle(si, splits):
    x = tiny(**SHAPES[si], seed=40 + si)
    assert kl.kl_decode_kernel_available(shape_of(x), kl.KL_KERNEL_TENSOR)
    out, err = decode(to_dev(x), shape_of(x), kernel=kl.KL_KERNEL_AUTO, num_splits=splits)
    assert err == 0
    assert_parity(out.cpu().numpy(), oracle_decode(x, _gpu.default_scale(x)),
                  f"{SHAPES[si]} S={splits}")


def test_large_group_many_splits_merge_in_kernel():
    # 40 splits: the last CTA of each head block merges through the staged path
    x = tiny(B=1, Hq=32, Hkv=1, D=128, P=16, lens=(9000,), seed=47)
    want = oracle_decode(x, _gpu.default_scale(x))
    for s in (8, 40):
        out, err = decode(to_dev(x), shape_of(x), num_splits=s)
        assert err == 0
        assert_parity(out.cpu().numpy(), want, f"S={s}")


def test_large_group_composed_query():
    """No W^R: the query already is the composed x W^Q W^R (three sibling CTAs)."""
    x = tiny(B=2, Hq=24, Hkv=1, D=128, P=16, lens=(700, 1900), seed=52)
    g = to_dev(x)
    sh = shape_of(x)
    out = torch.full((2, 24, 128), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, 3)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_attention_ex(sh, g["q"], None, g["v_cache"], g["block_table"], g["seq_lens"],
                              kl.decode_options(3, kl.KL_KERNEL_TENSOR), out, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    y = dict(x)
    y["w_r"] = torch.eye(128, dtype=torch.float32).expand(1, 128, 128).contiguous().to(torch.bfloat16)
    assert_parity(out.cpu().numpy(), oracle_decode(y, _gpu.default_scale(x)), "composed query")


def test_large_group_per_query_head_routing():
    x = tiny(B=2, Hq=128, Hkv=8, D=128, P=16, lens=(260, 999), wr_per_query_head=True, seed=48)
    out, err = decode(to_dev(x), shape_of(x), num_splits=2)
    assert err == 0
    assert_parity(out.cpu().numpy(), oracle_decode(x, _gpu.default_scale(x)), "per-head W^R")


def test_large_group_split_states():
    x = tiny(B=2, Hq=32, Hkv=1, D=128, P=16, lens=(1500, 300), seed=49)
    g = to_dev(x)
    sh = shape_of(x)
    S = kl.kl_decode_num_splits(sh, 3)
    B, Hq, D = x["q"].shape
    po = torch.full((B, Hq, S, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    pml = torch.full((B, Hq, S, 2), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    kl.kl_decode_attention_ex(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"], g["seq_lens"],
                              kl.decode_options(3, kl.KL_KERNEL_TENSOR, po, pml), None,
                              kl.KL_FP32, None, err)
    out = torch.full((B, Hq, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    kl.kl_combine(sh, po, pml, S, out, kl.KL_FP32)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert_parity(out.cpu().numpy(), oracle_decode(x, _gpu.default_scale(x)), "states merged")


def test_large_group_split_states_several_per_cta():
    """The most splits of one sequence (235 of 128 tokens): two sibling CTAs per split would
    overflow a wave, so each CTA runs two consecutive splits and writes a state for each; every
    state against the oracle's, and their merge against the whole decode."""
    x = tiny(B=1, Hq=16, Hkv=1, D=128, P=16, lens=(30000,), seed=53)
    g = to_dev(x)
    sh = shape_of(x)
    S = kl.kl_decode_num_splits(sh, 1000)
    B, Hq, D = x["q"].shape
    po = torch.full((B, Hq, S, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    pml = torch.full((B, Hq, S, 2), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    kl.kl_decode_attention_ex(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"], g["seq_lens"],
                              kl.decode_options(1000, kl.KL_KERNEL_TENSOR, po, pml), None,
                              kl.KL_FP32, None, err)
    out = torch.full((B, Hq, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    kl.kl_combine(sh, po, pml, S, out, kl.KL_FP32)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert_parity(out.cpu().numpy(), oracle_decode(x, _gpu.default_scale(x)), "states merged")
    lmax = x["block_table"].shape[1] * 16
    chunk = -(-(-(-lmax // S)) // 128) * 128        # ceil(lmax / S), rounded up to 128
    want_o, want_ml = oracle.decode_partial(bf16_bits(x["q"]), bf16_bits(x["w_r"]),
                                            bf16_bits(x["v_cache"]), x["block_table"].numpy(),
                                            x["seq_lens"].numpy(), scale=_gpu.default_scale(x),
                                            chunk=chunk, num_splits=S)
    got_o, got_ml = po.cpu().numpy().astype(np.float64), pml.cpu().numpy().astype(np.float64)
    full = want_ml[..., 1] > 0
    assert np.array_equal(got_ml[..., 1] > 0, full), "empty splits differ"
    assert_parity(got_o[full], want_o[full], f"split states S={S}")
    m_g, m_w = got_ml[..., 0][full], want_ml[..., 0][full]
    assert np.all(np.abs(m_g - m_w) <= 1e-3 + 1e-4 * np.abs(m_w)), "largest scores differ"


@pytest.mark.parametrize("splits", [1, 3, 0])
def test_large_group_fused_step(splits):
    x = tiny(B=2, Hq=128, Hkv=8, D=128, P=16, lens=(700, 1290), seed=50)
    g = to_dev(x)
    sh = shape_of(x)
    B, Hq, D = x["q"].shape
    out = torch.full((B, Hq, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_step(sh, g["q"], g["w_r"], g["v_new"], g["positions"], g["v_cache"],
                      g["block_table"], g["seq_lens"], kl.decode_options(splits), out,
                      kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    cache = oracle.append(bf16_bits(x["v_cache"]), bf16_bits(x["v_new"]), x["block_table"].numpy(),
                          x["positions"].numpy())
    np.testing.assert_array_equal(bf16_bits(g["v_cache"].cpu()), cache)
    y = dict(x)
    y["v_cache"] = torch.from_numpy(cache.view(np.int16)).view(torch.bfloat16)
    assert_parity(out.cpu().numpy(), oracle_decode(y, _gpu.default_scale(x)), f"S={splits}")


def test_large_group_standard_kv_decode():
    x = tiny(B=2, Hq=32, Hkv=1, D=128, P=16, lens=(300, 1111), seed=51)
    kc = torch.randn(x["v_cache"].shape, generator=torch.Generator().manual_seed(4)).to(torch.bfloat16)
    out, err = decode(to_dev(x), shape_of(x), num_splits=2, k_cache=kc.to(_gpu.dev()))
    assert err == 0
    want = oracle.standard_decode(bf16_bits(x["q"]), bf16_bits(kc), bf16_bits(x["v_cache"]),
                                  x["block_table"].numpy(), x["seq_lens"].numpy(),
                                  scale=_gpu.default_scale(x))
    assert_parity(out.cpu().numpy(), want, "standard K+V, MQA 32")


@pytest.mark.parametrize("si", [0, 1, 2])
@pytest.mark.parametrize("splits", [1, 3, 0])
def test_large_group_fp8_decode(si, splits):
    x = tiny(**SHAPES[si], seed=60 + si)
    codes, scales = oracle.quantize_rows(bf16_bits(x["v_cache"]))
    g = to_dev(x)
    sh = shape_of(x)
    B, Hq, D = x["q"].shape
    out = torch.full((B, Hq, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_attention_fp8(sh, g["q"], g["w_r"], torch.from_numpy(codes).to(_gpu.dev()),
                               torch.from_numpy(scales).to(_gpu.dev()), g["block_table"],
                               g["seq_lens"], splits, out, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    want = oracle.decode_fp8(bf16_bits(x["q"]), bf16_bits(x["w_r"]), codes, scales,
                             x["block_table"].numpy(), x["seq_lens"].numpy(),
                             scale=1.0 / math.sqrt(D))
    assert_parity(out.cpu().numpy(), want, f"fp8 {SHAPES[si]} S={splits}")


def test_cuda_core_kernel_rejects_large_groups():
    x = tiny(B=1, Hq=16, Hkv=1, D=128, P=16, lens=(100,))
    assert not kl.kl_decode_kernel_available(shape_of(x), kl.KL_KERNEL_SIMT)
    with pytest.raises(kl.KLError) as e:
        decode(to_dev(x), shape_of(x), kernel=kl.KL_KERNEL_SIMT, num_splits=1)
    assert e.value.status == kl.KL_ERR_UNSUPPORTED
