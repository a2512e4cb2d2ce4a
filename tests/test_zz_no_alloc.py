"""kl_decode_attention_noalloc: the decode for callers that cannot allocate device memory.

Such callers (a plugin inside a framework that owns all device memory, a latency-critical
path that cannot take an allocation's synchronization) pass inputs and outputs only; the
split states go to the library's fixed device scratch. Here its output is checked against
kl_decode_attention's (which uses a caller workspace) on two calls in a row, at the parity
tolerance of the other GPU tests. This file is collected last on purpose.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300.workloads import WORKLOADS, generate
from tests._gpu import ATOL, RTOL, shape_of, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


def _reference(g, sh, splits):
    out = torch.empty(g["q"].shape, dtype=torch.float32, device="cuda")
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, splits)), dtype=torch.uint8,
                     device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    kl.kl_decode_attention(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"], g["seq_lens"],
                           splits, out, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return out.cpu().numpy()


@pytest.mark.parametrize("name,splits", [("small_gqa", 5), ("tiny_mha", 2)])
def test_noalloc_matches_workspace_decode_twice(name, splits):
    x = generate(WORKLOADS[name])
    g = to_dev(x)
    sh = shape_of(x)
    assert kl.kl_decode_num_splits(sh, splits) > 1          # the scratch is really used
    want = _reference(g, sh, splits)
    for _ in range(2):
        out = torch.full(g["q"].shape, float("nan"), dtype=torch.float32, device="cuda")
        err = torch.zeros(1, dtype=torch.int32, device="cuda")
        kl.kl_decode_attention_noalloc(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                                       g["seq_lens"], splits, out, kl.KL_FP32, err)
        torch.cuda.synchronize()
        assert int(err.item()) == 0
        got = out.cpu().numpy()
        bad = ~(np.abs(got - want) <= ATOL + RTOL * np.abs(want))
        assert not bad.any(), f"{int(bad.sum())} outputs differ"


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
