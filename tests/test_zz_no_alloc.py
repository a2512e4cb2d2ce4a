"""kl_decode_attention_noalloc: the decode for callers that cannot allocate device memory.

Such callers (a plugin inside a framework that owns all device memory, a latency-critical
path that cannot take an allocation's synchronization) pass inputs and outputs only; the
split states go to the library's fixed device scratch. Here its output is checked against the
fp64 oracle and against kl_decode_attention's (which uses a caller workspace) on two calls in a
row, at the parity tolerance of the other GPU tests; a call with a bad block-table entry must
report it, and a clean call right after it, over the scratch that call left behind, must be
right again. This file is collected last on purpose.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300.workloads import WORKLOADS, generate
from tests._gpu import ATOL, RTOL, assert_parity, default_scale, oracle_decode, shape_of, to_dev
from tests._inputs import tiny

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


def _workspace_decode(g, sh, splits):
    out = torch.empty(g["q"].shape, dtype=torch.float32, device="cuda")
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, splits)), dtype=torch.uint8,
                     device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    kl.kl_decode_attention(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"], g["seq_lens"],
                           splits, out, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return out.cpu().numpy()


def _noalloc(g, sh, splits):
    out = torch.full(g["q"].shape, float("nan"), dtype=torch.float32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    kl.kl_decode_attention_noalloc(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                                   g["seq_lens"], splits, out, kl.KL_FP32, err)
    torch.cuda.synchronize()
    return out.cpu().numpy(), int(err.item())


@pytest.mark.parametrize("name,splits", [("small_gqa", 5), ("tiny_mha", 2)])
def test_noalloc_matches_oracle_and_workspace_decode_twice(name, splits):
    x = generate(WORKLOADS[name])
    g = to_dev(x)
    sh = shape_of(x)
    assert kl.kl_decode_num_splits(sh, splits) > 1          # the scratch is really used
    want = oracle_decode(x, default_scale(x))
    ws_out = _workspace_decode(g, sh, splits)
    for call in range(2):
        got, err = _noalloc(g, sh, splits)
        assert err == 0
        assert_parity(got, want, f"{name} noalloc call {call}")
        bad = ~(np.abs(got - ws_out) <= ATOL + RTOL * np.abs(ws_out))
        assert not bad.any(), f"{int(bad.sum())} outputs differ from the workspace decode"


def test_noalloc_reports_a_bad_page_then_a_clean_call_is_right():
    x = tiny(B=3, Hq=16, Hkv=4, D=128, P=16, lens=(300, 500, 700))
    sh = shape_of(x)
    splits = 3
    assert kl.kl_decode_num_splits(sh, splits) > 1
    want = oracle_decode(x, default_scale(x))
    y = dict(x)
    y["block_table"] = x["block_table"].clone()
    y["block_table"][0, 2] = x["num_pages"]                  # one page id past the pool
    got, err = _noalloc(to_dev(y), sh, splits)
    assert err & kl.KL_FLAG_BAD_PAGE
    assert_parity(got[1:], want[1:], "the sequences without the bad page")
    # a clean call over the split states the flagged call left in the scratch
    got, err = _noalloc(to_dev(x), sh, splits)
    assert err == 0
    assert_parity(got, want, "clean call after a flagged one")


def test_noalloc_rejects_split_states_beyond_the_scratch():
    x = generate(WORKLOADS["tiny_mha"])
    g = to_dev(x)
    # 4096 sequences x 64 heads x 8 splits x 130 floats is far beyond the fixed scratch
    big = kl.make_shape(4096, 64, 8, 128, 16, 16, 64)
    out = torch.empty(1, dtype=torch.float32, device="cuda")
    with pytest.raises(kl.KLError) as e:
        kl.kl_decode_attention_noalloc(big, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                                       g["seq_lens"], 8, out, kl.KL_FP32)
    assert e.value.status == kl.KL_ERR_WORKSPACE


def test_noalloc_rejects_an_unaligned_output():
    x = tiny(B=2, Hq=16, Hkv=4, D=128, P=16, lens=(300, 500))
    g = to_dev(x)
    sh = shape_of(x)
    buf = torch.empty(2 * 16 * 128 + 4, dtype=torch.float32, device="cuda")
    with pytest.raises(kl.KLError) as e:
        kl.kl_decode_attention_noalloc(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                                       g["seq_lens"], 3, buf.data_ptr() + 4, kl.KL_FP32)
    assert e.value.status == kl.KL_ERR_INVALID_ARG
