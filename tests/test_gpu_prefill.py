"""GPU parity of the chunked keyless prefill (and the chunk append) against the fp64 oracle.

Bar: the chunk append is bit-exact, page permutations leave the output bit-identical, and
every output element satisfies |gpu - oracle| <= 2e-3 + 1e-2 |oracle| (fp32 output; bf16 output
adds its own rounding, 2^-8 relative).
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
from tests._gpu import assert_parity, to_dev
from tests._inputs import tiny_prefill

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


def shape_of(x: dict, scale: float = 0.0) -> kl.kl_shape:
    num_pages, Hkv, P, D = x["v_cache"].shape
    B = x["seq_lens"].shape[0]
    Hq = x["q"].shape[1]
    return kl.make_shape(B, Hq, Hkv, D, P, num_pages, x["block_table"].shape[1],
                         x["workload"].wr_per_query_head, scale)


def run_prefill(x: dict, *, out_dtype=kl.KL_FP32, scale: float = 0.0, max_q=None):
    g = to_dev(x)
    T, Hq, D = x["q"].shape
    dt = torch.float32 if out_dtype == kl.KL_FP32 else torch.bfloat16
    out = torch.full((max(T, 1), Hq, D), float("nan"), dtype=dt, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    mq = int(x["q_lens"].max()) if max_q is None else max_q
    kl.kl_prefill_attention(shape_of(x, scale), g["q"], g["w_r"], g["v_cache"], g["block_table"],
                            g["seq_lens"], g["cu_q"], T, mq, out, out_dtype, err)
    torch.cuda.synchronize()
    return out[:T], int(err.item())


def oracle_prefill(x: dict, scale: float, rows=None):
    return oracle.prefill(bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"]),
                          x["block_table"].numpy(), x["seq_lens"].numpy(), x["cu_q"].numpy(),
                          scale=scale, wr_per_query_head=bool(x["workload"].wr_per_query_head),
                          rows=rows)


SHAPES = [
    # GQA group 4: a whole prompt, a chunk over a cached prefix, a single row (decode-like)
    dict(B=3, Hq=32, Hkv=8, D=128, P=16, lens=(300, 1000, 129), q_lens=(300, 200, 1)),
    # MHA, whole prompts of exactly one and several tiles, P 32
    dict(B=2, Hq=4, Hkv=4, D=128, P=32, lens=(128, 1024), q_lens=(128, 1024)),
    # Qwen2-1.5B heads (12 / 2, group 6), P 64, ragged
    dict(B=2, Hq=12, Hkv=2, D=128, P=64, lens=(777, 5), q_lens=(250, 5)),
    # MQA, P 128, an empty chunk next to a chunk that starts mid-page
    dict(B=3, Hq=8, Hkv=1, D=128, P=128, lens=(40, 0, 515), q_lens=(0, 0, 387)),
]


@pytest.mark.parametrize("shape", SHAPES)
def test_prefill_matches_oracle(shape):
    x = tiny_prefill(**shape, seed=31)
    scale = 1.0 / math.sqrt(shape["D"])
    got, err = run_prefill(x)
    assert err == 0
    want = oracle_prefill(x, scale)
    assert_parity(got.cpu().numpy(), want, f"prefill {shape}")


def test_prefill_per_query_head_routing_and_scale():
    x = tiny_prefill(B=2, Hq=16, Hkv=4, D=128, P=16, lens=(600, 333), q_lens=(600, 100),
                     wr_per_query_head=True, seed=32)
    got, err = run_prefill(x, scale=0.05)
    assert err == 0
    assert_parity(got.cpu().numpy(), oracle_prefill(x, 0.05), "per-query-head W^R, scale 0.05")


def test_prefill_bf16_output():
    x = tiny_prefill(B=2, Hq=8, Hkv=2, D=128, P=16, lens=(513, 64), q_lens=(200, 64), seed=33)
    got, err = run_prefill(x, out_dtype=kl.KL_BF16)
    assert err == 0
    want = oracle_prefill(x, 1.0 / math.sqrt(128))
    g = got.float().cpu().numpy().astype(np.float64)
    bad = np.abs(g - want) > 2e-3 + (1e-2 + 2.0 ** -8) * np.abs(want)
    assert not bad.any()


def test_long_prompt_sampled_rows():
    """A 4096-token prompt (32 cache tiles): every 37th row of every head against the oracle."""
    x = tiny_prefill(B=1, Hq=8, Hkv=2, D=128, P=16, lens=(4096,), q_lens=(4096,), seed=34)
    got, err = run_prefill(x)
    assert err == 0
    rows = [(r, h) for r in range(0, 4096, 37) for h in range(8)] + [(4095, h) for h in range(8)]
    want = oracle_prefill(x, 1.0 / math.sqrt(128), rows=rows)
    g = got.cpu().numpy()
    assert_parity(np.stack([g[r, h] for r, h in rows]), want, "4096-token prompt")


def test_large_scores_rescale_path():
    """Scores spanning tens of units in base 2 (W^R scaled up) drive the reference-maximum
    updates and the TMEM rescale of O many times per row."""
    x = tiny_prefill(B=2, Hq=8, Hkv=2, D=128, P=32, lens=(1500, 700), q_lens=(1500, 350), seed=35)
    x["w_r"] = (x["w_r"].float() * 6.0).to(torch.bfloat16)
    got, err = run_prefill(x)
    assert err == 0
    want = oracle_prefill(x, 1.0 / math.sqrt(128))
    assert_parity(got.cpu().numpy(), want, "large scores")


def test_page_permutation_is_bit_exact():
    x = tiny_prefill(B=2, Hq=8, Hkv=2, D=128, P=16, lens=(700, 260), q_lens=(300, 260), seed=36)
    a, e1 = run_prefill(x)
    perm = torch.randperm(x["v_cache"].shape[0], generator=torch.Generator().manual_seed(3))
    y = dict(x)
    y["v_cache"] = torch.empty_like(x["v_cache"])
    y["v_cache"][perm] = x["v_cache"]
    bt = x["block_table"].clone()
    valid = bt >= 0
    bt[valid] = perm[bt[valid].long()].to(torch.int32)
    y["block_table"] = bt
    b, e2 = run_prefill(y)
    assert e1 == 0 and e2 == 0
    assert torch.equal(a, b)


def test_single_row_chunks_match_oracle_decode():
    """n_b = 1 is a decode step: the prefill kernel's answer against the decode oracle."""
    x = tiny_prefill(B=4, Hq=16, Hkv=4, D=128, P=16, lens=(1, 17, 1000, 4097), q_lens=(1, 1, 1, 1),
                     seed=37)
    got, err = run_prefill(x)
    assert err == 0
    want = oracle.decode(bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"]),
                         x["block_table"].numpy(), x["seq_lens"].numpy(),
                         scale=1.0 / math.sqrt(128))
    assert_parity(got.cpu().numpy(), want, "one-row chunks")


def test_max_q_len_larger_than_needed_is_harmless():
    x = tiny_prefill(B=2, Hq=8, Hkv=2, D=128, P=16, lens=(300, 90), q_lens=(130, 90), seed=38)
    got, err = run_prefill(x, max_q=1000)
    assert err == 0
    assert_parity(got.cpu().numpy(), oracle_prefill(x, 1.0 / math.sqrt(128)), "max_q 1000")


def test_chunk_append_is_bit_exact():
    x = tiny_prefill(B=3, Hq=8, Hkv=2, D=128, P=16, lens=(5, 37, 100), q_lens=(5, 12, 1), seed=39)
    g = to_dev(x)
    T = int(x["cu_q"][-1])
    v_new = torch.randn(T, 2, 128, generator=torch.Generator().manual_seed(4)).to(torch.bfloat16)
    want = oracle.append_chunk(bf16_bits(x["v_cache"]), bf16_bits(v_new), x["block_table"].numpy(),
                               x["seq_lens"].numpy(), x["cu_q"].numpy())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    kl.kl_append_v_chunk(shape_of(x), v_new.to(_gpu.dev()), g["block_table"], g["seq_lens"],
                         g["cu_q"], T, 12, g["v_cache"], err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert np.array_equal(bf16_bits(g["v_cache"].cpu()), want)


def test_append_then_prefill_equals_oracle_on_the_appended_cache():
    x = tiny_prefill(B=2, Hq=8, Hkv=2, D=128, P=32, lens=(400, 129), q_lens=(144, 129), seed=40)
    g = to_dev(x)
    T = int(x["cu_q"][-1])
    v_new = torch.randn(T, 2, 128, generator=torch.Generator().manual_seed(5)).to(torch.bfloat16)
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    sh = shape_of(x)
    kl.kl_append_v_chunk(sh, v_new.to(_gpu.dev()), g["block_table"], g["seq_lens"], g["cu_q"], T,
                         144, g["v_cache"], err)
    out = torch.empty(T, 8, 128, dtype=torch.float32, device=_gpu.dev())
    kl.kl_prefill_attention(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"], g["seq_lens"],
                            g["cu_q"], T, 144, out, kl.KL_FP32, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    y = dict(x)
    y["v_cache"] = g["v_cache"].cpu()
    assert_parity(out.cpu().numpy(), oracle_prefill(y, 1.0 / math.sqrt(128)), "append + prefill")


def test_bad_lengths_and_pages_raise_flags():
    x = tiny_prefill(B=2, Hq=8, Hkv=2, D=128, P=16, lens=(64, 64), q_lens=(64, 64), seed=41)
    y = dict(x)
    y["seq_lens"] = torch.tensor([64, 10], dtype=torch.int32)     # n_1 = 64 > L_1 = 10
    _, err = run_prefill(y)
    assert err & kl.KL_FLAG_BAD_LENGTH
    z = dict(x)
    bt = x["block_table"].clone()
    bt[0, 1] = 10_000
    z["block_table"] = bt
    _, err = run_prefill(z)
    assert err & kl.KL_FLAG_BAD_PAGE


def test_outlier_values():
    """1 % of the cached entries scaled x20 (the ragged serving recipe): the case where the fp16
    weights of the output sum come closest to the bound."""
    x = tiny_prefill(B=2, Hq=8, Hkv=2, D=128, P=16, lens=(700, 260), q_lens=(300, 260), seed=36)
    v = x["v_cache"].float()
    mask = torch.rand(v.shape, generator=torch.Generator().manual_seed(9)) < 0.01
    x["v_cache"] = torch.where(mask, v * 20, v).to(torch.bfloat16)
    got, err = run_prefill(x)
    assert err == 0
    assert_parity(got.cpu().numpy(), oracle_prefill(x, 1.0 / math.sqrt(128)), "outliers")


def test_values_at_the_edge_of_fp16_and_beyond():
    """The output sum carries the cached values in fp16: the largest bf16 value it holds (65280)
    gives the oracle's answer, and a larger finite one (69632) makes outputs non-finite, which
    raises KL_FLAG_RANGE."""
    x = tiny_prefill(B=2, Hq=8, Hkv=2, D=128, P=16, lens=(300, 140), q_lens=(300, 140), seed=43)
    page = int(x["block_table"][0, 2])
    y = dict(x)
    y["v_cache"] = x["v_cache"].clone()
    y["v_cache"][page, 1, 5, 17] = -65280.0
    y["v_cache"][page, 0, 9, 100] = 65280.0
    got, err = run_prefill(y)
    assert err == 0
    assert_parity(got.cpu().numpy(), oracle_prefill(y, 1.0 / math.sqrt(128)), "65280")
    z = dict(x)
    z["v_cache"] = x["v_cache"].clone()
    z["v_cache"][page, 0, 9, 100] = 69632.0
    _, err = run_prefill(z)
    assert err & kl.KL_FLAG_RANGE


def test_head_dim_64_is_unsupported():
    x = tiny_prefill(B=1, Hq=4, Hkv=4, D=64, P=16, lens=(32,), q_lens=(32,), seed=42)
    with pytest.raises(kl.KLError) as e:
        run_prefill(x)
    assert e.value.status == kl.KL_ERR_UNSUPPORTED
