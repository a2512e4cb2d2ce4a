"""GPU parity of the decode over a latent value-only cache (absorbed query, tensor-core decode
over the latent rows, output expansion) against the fp64 oracle, through the C ABI.
Bar: |gpu - oracle| <= 2e-3 + 1e-2 |oracle| elementwise (fp32 output; bf16 adds 2^-8)."""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300.workloads import WORKLOADS, bf16_bits, generate
from tests import _gpu
from tests._gpu import assert_parity, to_dev
from tests._inputs import tiny_latent

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


def lshape(x, scale=0.0):
    num_pages, Hl, P, r = x["v_lat"].shape
    B, Hq, D = x["q"].shape
    return kl.make_latent_shape(B, Hq, Hl, D, r, P, num_pages, x["block_table"].shape[1],
                                x["workload"].wr_per_query_head, scale)


def run_latent(x, *, num_splits=0, out_dtype=kl.KL_FP32, scale=0.0):
    g = to_dev(x)
    B, Hq, D = x["q"].shape
    sh = lshape(x, scale)
    dt = torch.float32 if out_dtype == kl.KL_FP32 else torch.bfloat16
    out = torch.full((B, Hq, D), float("nan"), dtype=dt, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_latent_workspace_size(sh, num_splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_latent_decode(sh, g["q"], g["w_r"], g["w_post"], g["v_lat"], g["block_table"],
                        g["seq_lens"], num_splits, out, out_dtype, ws, err)
    torch.cuda.synchronize()
    return out, int(err.item())


def oracle_latent(x, scale):
    return oracle.latent_decode(bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["w_post"]),
                                bf16_bits(x["v_lat"]), x["block_table"].numpy(),
                                x["seq_lens"].numpy(), scale=scale,
                                wr_per_query_head=bool(x["workload"].wr_per_query_head))


SHAPES = [
    dict(B=3, Hq=8, Hl=2, D=128, r=128, P=16, lens=(1, 37, 300)),     # group latents
    dict(B=2, Hq=8, Hl=1, D=64, r=128, P=32, lens=(513, 9)),          # one shared latent, D 64
    dict(B=4, Hq=32, Hl=4, D=128, r=128, P=16, lens=(0, 129, 1000, 2048)),
]


@pytest.mark.parametrize("si", range(len(SHAPES)))
@pytest.mark.parametrize("num_splits", [1, 3, 0])
def test_latent_decode_matches_oracle(si, num_splits):
    shape = SHAPES[si]
    x = tiny_latent(**shape, seed=61 + si)
    got, err = run_latent(x, num_splits=num_splits)
    assert err == 0
    assert_parity(got.cpu().numpy(), oracle_latent(x, 1.0 / math.sqrt(shape["r"])),
                  f"latent {shape} S={num_splits}")


def test_latent_per_query_head_routing_scale_and_bf16():
    x = tiny_latent(B=2, Hq=16, Hl=2, D=128, r=128, P=16, lens=(700, 64), wr_per_query_head=True,
                    seed=71)
    got, err = run_latent(x, scale=0.05, out_dtype=kl.KL_BF16)
    assert err == 0
    want = oracle_latent(x, 0.05)
    g = got.float().cpu().numpy().astype(np.float64)
    assert not (np.abs(g - want) > 2e-3 + (1e-2 + 2.0 ** -8) * np.abs(want)).any()


def test_latent_workspace_reuse_two_calls():
    x = tiny_latent(B=3, Hq=8, Hl=2, D=128, r=128, P=16, lens=(900, 2000, 31), seed=72)
    g = to_dev(x)
    sh = lshape(x)
    ws = torch.zeros(kl.kl_latent_workspace_size(sh, 0), dtype=torch.uint8, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    outs = []
    for _ in range(2):
        out = torch.empty(3, 8, 128, dtype=torch.float32, device=_gpu.dev())
        kl.kl_latent_decode(sh, g["q"], g["w_r"], g["w_post"], g["v_lat"], g["block_table"],
                            g["seq_lens"], 0, out, kl.KL_FP32, ws, err)
        outs.append(out)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert torch.equal(outs[0], outs[1])
    assert_parity(outs[0].cpu().numpy(), oracle_latent(x, 1.0 / math.sqrt(128)), "reuse")


def test_latent_unsupported_shapes():
    x = tiny_latent(B=1, Hq=8, Hl=2, D=128, r=64, lens=(10,), seed=73)
    assert kl.kl_latent_workspace_size(lshape(x), 0) == 0
    with pytest.raises(kl.KLError) as e:
        run_latent(x)
    assert e.value.status == kl.KL_ERR_UNSUPPORTED
    y = tiny_latent(B=1, Hq=32, Hl=2, D=128, r=128, lens=(10,), seed=74)   # 16 heads per group
    with pytest.raises(kl.KLError) as e:
        run_latent(y)
    assert e.value.status == kl.KL_ERR_UNSUPPORTED


def test_latent_two_sequence_blocks_with_a_ragged_tail():
    """130 sequences: the projection kernels run two 128-sequence blocks, the second with two
    rows (the rest of its TMA boxes read as zeros and are never stored)."""
    lens = tuple(int(v) for v in np.random.default_rng(75).integers(0, 200, 130))
    x = tiny_latent(B=130, Hq=8, Hl=2, D=128, r=128, P=16, lens=lens, seed=75)
    got, err = run_latent(x)
    assert err == 0
    assert_parity(got.cpu().numpy(), oracle_latent(x, 1.0 / math.sqrt(128)), "130 sequences")


@pytest.mark.parametrize("out_dtype", [kl.KL_BF16, kl.KL_FP32])
def test_latent_head_dim_64_outputs(out_dtype):
    """D 64: one 64-value half per query row, N = 64 expansion; bf16 rows are one 128-byte box,
    fp32 rows two."""
    x = tiny_latent(B=5, Hq=12, Hl=3, D=64, r=128, P=16, lens=(3, 250, 1, 77, 640), seed=76)
    got, err = run_latent(x, out_dtype=out_dtype)
    assert err == 0
    want = oracle_latent(x, 1.0 / math.sqrt(128))
    g = got.float().cpu().numpy().astype(np.float64)
    rel = 1e-2 + (2.0 ** -8 if out_dtype == kl.KL_BF16 else 0.0)
    assert not (np.abs(g - want) > 2e-3 + rel * np.abs(want)).any()


@pytest.mark.slow
def test_latent_serving_sampled_parity():
    """The full latent serving workload (64 sequences of 8192 tokens, 32 query heads over 4
    latent groups) in the bench's launch configuration; sampled heads against the oracle."""
    wl = WORKLOADS["latent_serving"]
    x = generate(wl)
    got, err = run_latent(x, num_splits=max(wl.num_splits, 0), out_dtype=kl.KL_BF16)
    assert err == 0
    rng = np.random.default_rng(wl.seed)
    B, Hq = wl.num_seqs, wl.num_q_heads
    heads = [(int(b), int(h)) for b, h in zip(rng.integers(0, B, 40), rng.integers(0, Hq, 40))]
    heads += [(B - 1, Hq - 1), (0, 0)]
    want = oracle.latent_decode(bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["w_post"]),
                                bf16_bits(x["v_lat"]), x["block_table"].numpy(),
                                x["seq_lens"].numpy(), scale=1.0 / math.sqrt(wl.latent_dim),
                                wr_per_query_head=bool(wl.wr_per_query_head), heads=heads)
    g = got.float().cpu().numpy().astype(np.float64)
    sampled = np.stack([g[b, h] for b, h in heads])
    assert not (np.abs(sampled - want) > 2e-3 + (1e-2 + 2.0 ** -8) * np.abs(want)).any()
    assert np.isfinite(g).all()


def test_latent_back_to_back_calls_with_different_queries():
    """Two calls on one stream, same workspace, different queries, no synchronization between
    them: the decode of each call must read that call's absorbed queries and its expansion that
    call's decode output (a dependent launch that read too early would return the other call's
    values)."""
    x = tiny_latent(B=6, Hq=16, Hl=2, D=128, r=128, P=16, lens=(1500, 2048, 77, 900, 1, 3000),
                    seed=77)
    y = dict(x)
    y["q"] = torch.randn(x["q"].shape, generator=torch.Generator().manual_seed(78)).to(torch.bfloat16)
    g = to_dev(x)
    q2 = y["q"].to(_gpu.dev())
    sh = lshape(x)
    ws = torch.zeros(kl.kl_latent_workspace_size(sh, 0), dtype=torch.uint8, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    outs = []
    for q in (g["q"], q2, g["q"], q2):
        out = torch.empty(6, 16, 128, dtype=torch.float32, device=_gpu.dev())
        kl.kl_latent_decode(sh, q, g["w_r"], g["w_post"], g["v_lat"], g["block_table"],
                            g["seq_lens"], 0, out, kl.KL_FP32, ws, err)
        outs.append(out)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    scale = 1.0 / math.sqrt(128)
    want1, want2 = oracle_latent(x, scale), oracle_latent(y, scale)
    for i, out in enumerate(outs):
        assert_parity(out.cpu().numpy(), want1 if i % 2 == 0 else want2, f"call {i}")


def test_latent_decode_step_appends_then_decodes():
    """kl_latent_decode_step: the current token's latent rows land bit-exactly where the oracle's
    append puts them, the output matches the oracle over the appended cache, and it is
    bit-identical to a separate kl_append_v followed by kl_latent_decode."""
    x = tiny_latent(B=4, Hq=16, Hl=2, D=128, r=128, P=16, lens=(1, 40, 700, 1500), seed=79)
    B, Hq, D = x["q"].shape
    num_pages, Hl, P, r = x["v_lat"].shape
    v_new = torch.randn(B, Hl, r, generator=torch.Generator().manual_seed(80)).to(torch.bfloat16)
    positions = (x["seq_lens"] - 1).to(torch.int32)
    sh = lshape(x)
    ws = torch.zeros(max(256, kl.kl_latent_workspace_size(sh, 0)), dtype=torch.uint8,
                     device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    g = to_dev(x)
    vn, pos = v_new.to(_gpu.dev()), positions.to(_gpu.dev())
    out = torch.empty(B, Hq, D, dtype=torch.float32, device=_gpu.dev())
    kl.kl_latent_decode_step(sh, g["q"], g["w_r"], g["w_post"], vn, pos, g["v_lat"],
                             g["block_table"], g["seq_lens"], 0, out, kl.KL_FP32, ws, err)
    # the unfused pair on a second copy of the cache
    v2 = to_dev(x)["v_lat"]
    ash = kl.make_shape(B, Hq, Hl, r, P, num_pages, x["block_table"].shape[1])
    kl.kl_append_v(ash, vn, g["block_table"], pos, v2, err)
    out2 = torch.empty_like(out)
    kl.kl_latent_decode(sh, g["q"], g["w_r"], g["w_post"], v2, g["block_table"], g["seq_lens"],
                        0, out2, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    want_cache = oracle.append(bf16_bits(x["v_lat"]), bf16_bits(v_new), x["block_table"].numpy(),
                               positions.numpy())
    assert np.array_equal(bf16_bits(g["v_lat"].cpu()), want_cache)
    assert torch.equal(out, out2)
    y = dict(x)
    y["v_lat"] = torch.from_numpy(want_cache.view(np.int16)).view(torch.bfloat16)
    assert_parity(out.cpu().numpy(), oracle_latent(y, 1.0 / math.sqrt(r)), "latent step")
