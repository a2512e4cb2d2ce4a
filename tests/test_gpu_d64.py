"""GPU parity of the tensor-core decode at head dim 64 (GPT-2's head layout, the paper's main
experiments in Section 5): every cached row read once for score and output, against the fp64
oracle at |gpu - oracle| <= 2e-3 + 1e-2 |oracle|, appended rows and permutations bit-exact.

With an even number of value heads and groups of up to 4 query heads, one CTA takes two value
heads side by side in its 128-wide tiles (block-diagonal routing); otherwise a 64-dim row fills
half of a zero-padded tile. Both layouts are covered below.
"""
from __future__ import annotations

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

TC = kl.KL_KERNEL_TENSOR


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


SHAPES = [
    dict(B=2, Hq=12, Hkv=12, D=64, P=16, lens=(1024, 33)),        # GPT-2 small heads (MHA)
    dict(B=3, Hq=32, Hkv=8, D=64, P=32, lens=(0, 129, 2000)),     # GQA 4, P 32
    dict(B=2, Hq=64, Hkv=8, D=64, P=16, lens=(700, 1500)),        # GQA 8
    dict(B=1, Hq=16, Hkv=1, D=64, P=64, lens=(3000,)),            # MQA, group 16 (two CTAs)
    dict(B=2, Hq=6, Hkv=3, D=64, P=16, lens=(800, 5)),            # odd value-head count
]


@pytest.mark.parametrize("si", range(len(SHAPES)))
@pytest.mark.parametrize("splits", [1, 3, 0, 40])
def test_d64_decode_matches_oracle(si, splits):
    x = tiny(**SHAPES[si], seed=80 + si)
    assert kl.kl_decode_kernel_available(shape_of(x), TC)
    out, err = decode(to_dev(x), shape_of(x), kernel=TC, num_splits=splits)
    assert err == 0
    assert_parity(out.cpu().numpy(), oracle_decode(x, _gpu.default_scale(x)),
                  f"{SHAPES[si]} S={splits}")


def test_d64_per_query_head_routing_custom_scale_bf16_output():
    x = tiny(B=2, Hq=16, Hkv=4, D=64, P=16, lens=(300, 901), wr_per_query_head=True, seed=85)
    sh = shape_of(x, scale=0.2)
    out32, err = decode(to_dev(x), sh, kernel=TC, num_splits=2)
    assert err == 0
    out16, _ = decode(to_dev(x), sh, kernel=TC, num_splits=2, out_dtype=kl.KL_BF16)
    assert_parity(out32.cpu().numpy(), oracle_decode(x, 0.2), "per-head W^R, scale 0.2")
    np.testing.assert_allclose(out16.float().cpu().numpy(), out32.cpu().numpy(), rtol=2 ** -8,
                               atol=1e-6)


def test_d64_composed_query():
    """No W^R: the query already is the composed x W^Q W^R; the oracle with W^R = I."""
    x = tiny(B=2, Hq=8, Hkv=2, D=64, P=16, lens=(500, 77), seed=86)
    g = to_dev(x)
    sh = shape_of(x)
    out = torch.full((2, 8, 64), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, 3)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_attention_ex(sh, g["q"], None, g["v_cache"], g["block_table"], g["seq_lens"],
                              kl.decode_options(3, TC), out, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    y = dict(x)
    y["w_r"] = torch.eye(64, dtype=torch.float32).expand(2, 64, 64).contiguous().to(torch.bfloat16)
    assert_parity(out.cpu().numpy(), oracle_decode(y, _gpu.default_scale(x)), "composed query")


@pytest.mark.parametrize("splits", [1, 3, 0])
def test_d64_fused_step(splits):
    x = tiny(B=3, Hq=16, Hkv=4, D=64, P=16, lens=(40, 600, 1300), seed=87)
    x["positions"] = torch.tensor([39, 300, 1299], dtype=torch.int32)   # last, middle, last
    g = to_dev(x)
    sh = shape_of(x)
    out = torch.full((3, 16, 64), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_step(sh, g["q"], g["w_r"], g["v_new"], g["positions"], g["v_cache"],
                      g["block_table"], g["seq_lens"], kl.decode_options(splits, TC), out,
                      kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    cache = oracle.append(bf16_bits(x["v_cache"]), bf16_bits(x["v_new"]), x["block_table"].numpy(),
                          x["positions"].numpy())
    np.testing.assert_array_equal(bf16_bits(g["v_cache"].cpu()), cache)
    y = dict(x)
    y["v_cache"] = torch.from_numpy(cache.view(np.int16)).view(torch.bfloat16)
    assert_parity(out.cpu().numpy(), oracle_decode(y, _gpu.default_scale(x)), f"S={splits}")


def test_d64_split_states():
    x = tiny(B=2, Hq=8, Hkv=2, D=64, P=16, lens=(2000, 300), seed=88)
    g = to_dev(x)
    sh = shape_of(x)
    for splits in (3, 64):
        S = kl.kl_decode_num_splits(sh, splits)
        po = torch.full((2, 8, S, 64), float("nan"), dtype=torch.float32, device=_gpu.dev())
        pml = torch.full((2, 8, S, 2), float("nan"), dtype=torch.float32, device=_gpu.dev())
        err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
        kl.kl_decode_attention_ex(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                                  g["seq_lens"], kl.decode_options(splits, TC, po, pml), None,
                                  kl.KL_FP32, None, err)
        torch.cuda.synchronize()
        assert int(err.item()) == 0
        lmax = x["block_table"].shape[1] * 16
        chunk = -(-(-(-lmax // S)) // 128) * 128        # ceil(lmax / S), rounded up to 128
        want_o, want_ml = oracle.decode_partial(bf16_bits(x["q"]), bf16_bits(x["w_r"]),
                                                bf16_bits(x["v_cache"]), x["block_table"].numpy(),
                                                x["seq_lens"].numpy(), scale=_gpu.default_scale(x),
                                                chunk=chunk, num_splits=S)
        got_o, got_ml = po.cpu().numpy().astype(np.float64), pml.cpu().numpy().astype(np.float64)
        full = want_ml[..., 1] > 0
        assert np.array_equal(got_ml[..., 1] > 0, full), "empty splits differ"
        assert np.all(np.isneginf(got_ml[..., 0][~full])) and np.all(got_o[~full] == 0.0)
        assert_parity(got_o[full], want_o[full], f"split states S={S}")
        m_g, m_w = got_ml[..., 0][full], want_ml[..., 0][full]
        assert np.all(np.abs(m_g - m_w) <= 1e-3 + 1e-4 * np.abs(m_w)), "largest scores differ"
        l_g, l_w = got_ml[..., 1][full], want_ml[..., 1][full]
        assert np.all(np.abs(l_g - l_w) <= 1e-3 * l_w), "exponent sums differ"


def test_d64_standard_kv_decode():
    x = tiny(B=2, Hq=16, Hkv=4, D=64, P=16, lens=(300, 1111), seed=89)
    kc = torch.randn(x["v_cache"].shape, generator=torch.Generator().manual_seed(9)).to(torch.bfloat16)
    out, err = decode(to_dev(x), shape_of(x), kernel=TC, num_splits=2, k_cache=kc.to(_gpu.dev()))
    assert err == 0
    want = oracle.standard_decode(bf16_bits(x["q"]), bf16_bits(kc), bf16_bits(x["v_cache"]),
                                  x["block_table"].numpy(), x["seq_lens"].numpy(),
                                  scale=_gpu.default_scale(x))
    assert_parity(out.cpu().numpy(), want, "standard K+V, head dim 64")


def test_d64_block_table_permutation_is_bit_exact():
    x = tiny(B=3, Hq=16, Hkv=4, D=64, P=16, lens=(100, 555, 1024), seed=90)
    out1, _ = decode(to_dev(x), shape_of(x), kernel=TC, num_splits=3)
    perm = torch.randperm(x["num_pages"], generator=torch.Generator().manual_seed(6))
    inv = torch.argsort(perm)
    y = dict(x)
    y["v_cache"] = x["v_cache"][perm].contiguous()
    bt = x["block_table"].clone()
    m = bt >= 0
    bt[m] = inv[bt[m].long()].to(torch.int32)
    y["block_table"] = bt
    out2, _ = decode(to_dev(y), shape_of(y), kernel=TC, num_splits=3)
    assert torch.equal(out1.cpu(), out2.cpu())
