"""Failure detection of the tensor-core decodes, tested without a GPU fault.

Every wait of a decode CTA on its own pipeline is bounded. With the library's wait limit set to
one nanosecond, the waits run out on purpose: the call must return, raise KL_FLAG_TIMEOUT in the
device error word, and leave the context usable -- a normal call right after it (the limit
restored, the workspace zero-filled again as the header asks) matches the fp64 oracle.
"""
from __future__ import annotations

import math

import pytest
import torch

import oracle
import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300.workloads import bf16_bits
from tests import _gpu
from tests._gpu import assert_parity, oracle_decode, shape_of, to_dev
from tests._inputs import tiny

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


class short_waits:
    """The decodes' pipeline waits limited to `ns` nanoseconds inside the block."""

    def __init__(self, ns: int):
        self.ns = ns

    def __enter__(self):
        self.prev = kl.kl_set_wait_timeout_ns(self.ns)

    def __exit__(self, *exc):
        kl.kl_set_wait_timeout_ns(0)


def test_wait_limit_setting_round_trips():
    default = kl.kl_set_wait_timeout_ns(0)
    assert default == 1_000_000_000
    assert kl.kl_set_wait_timeout_ns(5_000) == default
    assert kl.kl_set_wait_timeout_ns(0) == 5_000
    assert kl.kl_set_wait_timeout_ns(0) == default


@pytest.mark.parametrize("splits", [1, 4, 40])
@pytest.mark.parametrize("Hq", [32, 64, 128])
def test_bf16_decode_times_out_then_recovers(splits, Hq):
    x = tiny(B=2, Hq=Hq, Hkv=8, D=128, P=16, lens=(5000, 3000), seed=71)
    g = to_dev(x)
    sh = shape_of(x)
    B, _, D = x["q"].shape
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    out = torch.full((B, Hq, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    opts = kl.decode_options(splits, kl.KL_KERNEL_TENSOR)
    with short_waits(1):
        kl.kl_decode_attention_ex(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                                  g["seq_lens"], opts, out, kl.KL_FP32, ws, err)
        torch.cuda.synchronize()
    assert int(err.item()) & kl.KL_FLAG_TIMEOUT
    ws.zero_()
    err.zero_()
    kl.kl_decode_attention_ex(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                              g["seq_lens"], opts, out, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert_parity(out.cpu().numpy(), oracle_decode(x, _gpu.default_scale(x)), f"after S={splits}")


@pytest.mark.parametrize("splits", [1, 3])
def test_fp8_decode_times_out_then_recovers(splits):
    x = tiny(B=2, Hq=32, Hkv=8, D=128, P=16, lens=(5000, 3000), seed=72)
    codes, scales = oracle.quantize_rows(bf16_bits(x["v_cache"]))
    g = to_dev(x)
    sh = shape_of(x)
    B, Hq, D = x["q"].shape
    c = torch.from_numpy(codes).to(_gpu.dev())
    s = torch.from_numpy(scales).to(_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    out = torch.full((B, Hq, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    with short_waits(1):
        kl.kl_decode_attention_fp8(sh, g["q"], g["w_r"], c, s, g["block_table"], g["seq_lens"],
                                   splits, out, kl.KL_FP32, ws, err)
        torch.cuda.synchronize()
    assert int(err.item()) & kl.KL_FLAG_TIMEOUT
    ws.zero_()
    err.zero_()
    kl.kl_decode_attention_fp8(sh, g["q"], g["w_r"], c, s, g["block_table"], g["seq_lens"],
                               splits, out, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    want = oracle.decode_fp8(bf16_bits(x["q"]), bf16_bits(x["w_r"]), codes, scales,
                             x["block_table"].numpy(), x["seq_lens"].numpy(),
                             scale=1.0 / math.sqrt(D))
    assert_parity(out.cpu().numpy(), want, f"fp8 after S={splits}")
