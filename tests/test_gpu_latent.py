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
from paper_2606_21848_gb300.workloads import bf16_bits
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
