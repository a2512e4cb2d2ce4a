"""Full-size parity in the bench's launch configuration: the fused decode step (kl_decode_step,
and kl_decode_step_fp8 for the FP8 cache) on the whole workload, with the workload's split
count and bf16 output, checked on sampled sequences against the fp64 oracle.

The oracle runs over a compact pool holding only the sampled sequences' pages (block table
renumbered), with the current token's row appended by the oracle's own append (or quantizing
append); nothing the GPU produced is an oracle input. The appended rows in the GPU's cache are
checked bit-exact against the oracle's append.
"""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300.workloads import WORKLOADS, bf16_bits, generate
from tests import _gpu
from tests._gpu import assert_parity, shape_of, to_dev

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


def _sampled_sequences(wl, n=8):
    rng = np.random.default_rng(wl.seed + 101)
    pick = {0, wl.num_seqs - 1} | {int(b) for b in rng.integers(0, wl.num_seqs, 3 * n)}
    return sorted(pick)[:n]


def _compact(x, seqs):
    """The sampled sequences' inputs over a pool of only their pages: (q, w_r, v, table,
    lengths, positions, v_new), bf16 as bit patterns, table renumbered."""
    P = x["v_cache"].shape[2]
    bt_all, sl_all = x["block_table"].numpy(), x["seq_lens"].numpy()
    used = sorted({int(p) for b in seqs for p in bt_all[b, :(int(sl_all[b]) + P - 1) // P]})
    remap = {p: i for i, p in enumerate(used)}
    bt = np.full((len(seqs), bt_all.shape[1]), -1, np.int32)
    for i, b in enumerate(seqs):
        for j in range((int(sl_all[b]) + P - 1) // P):
            bt[i, j] = remap[int(bt_all[b, j])]
    v = np.ascontiguousarray(bf16_bits(x["v_cache"])[used])
    return (np.ascontiguousarray(bf16_bits(x["q"])[seqs]), bf16_bits(x["w_r"]), v, bt,
            sl_all[seqs].copy(), x["positions"].numpy()[seqs].copy(),
            np.ascontiguousarray(bf16_bits(x["v_new"])[seqs]))


@pytest.mark.parametrize("name", ["long_context", "ragged_serving", "high_concurrency_70b",
                                  "mqa_group32", "gqa_group16", "mha_d64"])
def test_fused_step_full_size_sampled(name):
    wl = WORKLOADS[name]
    x = generate(wl)
    seqs = _sampled_sequences(wl)
    q, w, v, bt, sl, pos, v_new = _compact(x, seqs)        # before the GPU step touches the cache
    g = to_dev(x)
    sh = shape_of(x)
    B, Hq, D = x["q"].shape
    S = wl.num_splits
    out = torch.full((B, Hq, D), float("nan"), dtype=torch.bfloat16, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, S)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_step(sh, g["q"], g["w_r"], g["v_new"], g["positions"], g["v_cache"],
                      g["block_table"], g["seq_lens"], kl.decode_options(S), out, kl.KL_BF16, ws,
                      err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    # the appended rows, bit-exact
    P = x["v_cache"].shape[2]
    bt_all = x["block_table"].numpy()
    cache = g["v_cache"]
    for b in seqs:
        p = int(x["positions"][b])
        row = cache[int(bt_all[b, p // P]), :, p % P, :].cpu()
        np.testing.assert_array_equal(bf16_bits(row), bf16_bits(x["v_new"][b]))
    v_app = oracle.append(v, v_new, bt, pos)
    want = oracle.decode(q, w, v_app, bt, sl, scale=1.0 / math.sqrt(D))
    got = out[seqs].float().cpu().numpy()
    assert_parity(got, want, f"{name} S={S}")


def test_fused_fp8_step_full_size_sampled():
    """The FP8 cache of the default batch: the GPU quantizes the whole cache and runs the
    quantizing fused step; the oracle quantizes the sampled sequences' pages itself."""
    wl = WORKLOADS["high_concurrency_70b"]
    x = generate(wl)
    seqs = _sampled_sequences(wl)
    q, w, v, bt, sl, pos, v_new = _compact(x, seqs)
    g = to_dev(x)
    sh = shape_of(x)
    B, Hq, D = x["q"].shape
    codes = torch.empty(g["v_cache"].shape, dtype=torch.uint8, device=_gpu.dev())
    scales = torch.empty(g["v_cache"].shape[:-1], dtype=torch.float32, device=_gpu.dev())
    kl.kl_quantize_cache_fp8(sh, g["v_cache"], codes, scales)
    del g["v_cache"]
    out = torch.full((B, Hq, D), float("nan"), dtype=torch.bfloat16, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, 0)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_step_fp8(sh, g["q"], g["w_r"], g["v_new"], g["positions"], codes, scales,
                          g["block_table"], g["seq_lens"], 0, out, kl.KL_BF16, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    c_codes, c_scales = oracle.quantize_rows(v)
    c_codes, c_scales = oracle.append_fp8(c_codes, c_scales, v_new, bt, pos)
    want = oracle.decode_fp8(q, w, c_codes, c_scales, bt, sl, scale=1.0 / math.sqrt(D))
    got = out[seqs].float().cpu().numpy()
    assert_parity(got, want, "fp8 high_concurrency_70b")
