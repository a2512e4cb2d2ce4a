"""GPU parity of the FP8 value cache (E4M3 codes, one fp32 scale per cached row): the
quantizing append and the cache quantizer are bit-exact against the oracle's quantization, and
the decode over the FP8 cache matches the oracle's decode over the same codes and scales within
|gpu - oracle| <= 2e-3 + 1e-2 |oracle| (fp32 output)."""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300.workloads import bf16_bits
from tests import _gpu
from tests._gpu import assert_parity, shape_of, to_dev
from tests._inputs import tiny

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


def fp8_cache(x):
    """Codes and scales of the workload's bf16 cache, quantized by the oracle."""
    return oracle.quantize_rows(bf16_bits(x["v_cache"]))


def run_fp8(x, codes, scales, *, num_splits=0, out_dtype=kl.KL_FP32, composed=False):
    g = to_dev(x)
    sh = shape_of(x)
    B, Hq, D = x["q"].shape
    dt = torch.float32 if out_dtype == kl.KL_FP32 else torch.bfloat16
    out = torch.full((B, Hq, D), float("nan"), dtype=dt, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, num_splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    c = torch.from_numpy(codes).to(_gpu.dev())
    s = torch.from_numpy(scales).to(_gpu.dev())
    kl.kl_decode_attention_fp8(sh, g["q"], None if composed else g["w_r"], c, s, g["block_table"],
                               g["seq_lens"], num_splits, out, out_dtype, ws, err)
    torch.cuda.synchronize()
    return out, int(err.item())


SHAPES = [
    dict(B=3, Hq=32, Hkv=8, D=128, P=16, lens=(0, 129, 1000)),
    dict(B=2, Hq=64, Hkv=8, D=128, P=32, lens=(513, 2047)),
    dict(B=2, Hq=8, Hkv=1, D=128, P=16, lens=(1500, 9)),
    dict(B=2, Hq=12, Hkv=2, D=128, P=64, lens=(2222, 640)),
    dict(B=3, Hq=24, Hkv=8, D=128, P=128, lens=(5, 300, 1025)),
]


@pytest.mark.parametrize("si", range(len(SHAPES)))
@pytest.mark.parametrize("num_splits", [1, 3, 0])
def test_fp8_decode_matches_oracle(si, num_splits):
    x = tiny(**SHAPES[si], seed=91 + si)
    codes, scales = fp8_cache(x)
    got, err = run_fp8(x, codes, scales, num_splits=num_splits)
    assert err == 0
    want = oracle.decode_fp8(bf16_bits(x["q"]), bf16_bits(x["w_r"]), codes, scales,
                             x["block_table"].numpy(), x["seq_lens"].numpy(),
                             scale=1.0 / math.sqrt(128))
    assert_parity(got.cpu().numpy(), want, f"fp8 {SHAPES[si]} S={num_splits}")


def test_fp8_decode_outliers_composed_query_and_bf16_output():
    x = tiny(B=2, Hq=32, Hkv=8, D=128, P=16, lens=(3000, 77), seed=97)
    v = x["v_cache"].float()
    mask = torch.rand(v.shape, generator=torch.Generator().manual_seed(1)) < 0.01
    x["v_cache"] = torch.where(mask, v * 20.0, v).to(torch.bfloat16)
    codes, scales = fp8_cache(x)
    got, err = run_fp8(x, codes, scales, composed=True, out_dtype=kl.KL_BF16)
    assert err == 0
    eye = np.broadcast_to(np.eye(128, dtype=np.float32)[None], (8, 128, 128))
    w_eye = bf16_bits(torch.from_numpy(eye.copy()).to(torch.bfloat16))
    want = oracle.decode_fp8(bf16_bits(x["q"]), w_eye, codes, scales, x["block_table"].numpy(),
                             x["seq_lens"].numpy(), scale=1.0 / math.sqrt(128))
    g = got.float().cpu().numpy().astype(np.float64)
    assert not (np.abs(g - want) > 2e-3 + (1e-2 + 2.0 ** -8) * np.abs(want)).any()


def test_fp8_append_and_cache_quantizer_are_bit_exact():
    x = tiny(B=4, Hq=16, Hkv=8, D=128, P=32, lens=(1, 32, 97, 300), seed=98)
    g = to_dev(x)
    sh = shape_of(x)
    c = torch.empty(x["v_cache"].shape, dtype=torch.uint8, device=_gpu.dev())
    s = torch.empty(x["v_cache"].shape[:-1], dtype=torch.float32, device=_gpu.dev())
    kl.kl_quantize_cache_fp8(sh, g["v_cache"], c, s)
    torch.cuda.synchronize()
    codes, scales = fp8_cache(x)
    assert np.array_equal(c.cpu().numpy(), codes)
    assert np.array_equal(s.cpu().numpy(), scales)
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    kl.kl_append_v_fp8(sh, g["v_new"], g["block_table"], g["positions"], c, s, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    wc, ws_ = oracle.append_fp8(codes, scales, bf16_bits(x["v_new"]), x["block_table"].numpy(),
                                x["positions"].numpy())
    assert np.array_equal(c.cpu().numpy(), wc)
    assert np.array_equal(s.cpu().numpy(), ws_)


def test_fp8_page_permutation_is_bit_exact():
    x = tiny(B=2, Hq=32, Hkv=8, D=128, P=16, lens=(900, 260), seed=99)
    codes, scales = fp8_cache(x)
    a, e1 = run_fp8(x, codes, scales, num_splits=2)
    perm = np.random.default_rng(2).permutation(codes.shape[0])
    c2, s2 = np.empty_like(codes), np.empty_like(scales)
    c2[perm], s2[perm] = codes, scales
    y = dict(x)
    bt = x["block_table"].clone()
    valid = bt >= 0
    bt[valid] = torch.from_numpy(perm)[bt[valid].long()].to(torch.int32)
    y["block_table"] = bt
    b, e2 = run_fp8(y, c2, s2, num_splits=2)
    assert e1 == 0 and e2 == 0
    assert torch.equal(a, b)


def test_fp8_unsupported_shapes():
    x = tiny(B=1, Hq=8, Hkv=2, D=128, P=16, lens=(64,), wr_per_query_head=True, seed=100)
    codes, scales = fp8_cache(x)
    with pytest.raises(kl.KLError) as e:
        run_fp8(x, codes, scales)
    assert e.value.status == kl.KL_ERR_UNSUPPORTED


@pytest.mark.parametrize("num_splits", [1, 3, 0])
def test_fp8_decode_step_appends_then_decodes(num_splits):
    """kl_decode_step_fp8: the current token's rows are quantized into the cache bit-exactly as
    the oracle's append does it, the output matches the oracle's FP8 decode over the appended
    cache, and it is bit-identical to kl_append_v_fp8 followed by kl_decode_attention_fp8. One
    position lies past its sequence's end (it is written, and not attended)."""
    x = tiny(B=4, Hq=32, Hkv=8, D=128, P=16, lens=(1, 130, 1000, 2049), seed=98)
    codes, scales = fp8_cache(x)
    B, Hq, D = x["q"].shape
    v_new = torch.randn(B, 8, D, generator=torch.Generator().manual_seed(99)).to(torch.bfloat16)
    positions = (x["seq_lens"] - 1).to(torch.int32)
    positions[1] = 140                                     # past L = 130, inside its last page
    g = to_dev(x)
    sh = shape_of(x)
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, num_splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    vn, pos = v_new.to(_gpu.dev()), positions.to(_gpu.dev())
    c1, s1 = torch.from_numpy(codes).to(_gpu.dev()), torch.from_numpy(scales).to(_gpu.dev())
    c2, s2 = c1.clone(), s1.clone()
    out1 = torch.full((B, Hq, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    out2 = torch.full_like(out1, float("nan"))
    kl.kl_decode_step_fp8(sh, g["q"], g["w_r"], vn, pos, c1, s1, g["block_table"], g["seq_lens"],
                          num_splits, out1, kl.KL_FP32, ws, err)
    kl.kl_append_v_fp8(sh, vn, g["block_table"], pos, c2, s2, err)
    kl.kl_decode_attention_fp8(sh, g["q"], g["w_r"], c2, s2, g["block_table"], g["seq_lens"],
                               num_splits, out2, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    want_c, want_s = oracle.append_fp8(codes, scales, bf16_bits(v_new), x["block_table"].numpy(),
                                       positions.numpy())
    assert np.array_equal(c1.cpu().numpy(), want_c)
    assert np.array_equal(s1.cpu().numpy().view(np.uint32), want_s.view(np.uint32))
    assert torch.equal(out1, out2)
    want = oracle.decode_fp8(bf16_bits(x["q"]), bf16_bits(x["w_r"]), want_c, want_s,
                             x["block_table"].numpy(), x["seq_lens"].numpy(),
                             scale=1.0 / math.sqrt(128))
    assert_parity(out1.cpu().numpy(), want, f"fp8 step S={num_splits}")


def test_fp8_decode_step_flags_bad_position_and_page():
    """A negative position raises KL_FLAG_BAD_POSITION and a row whose page id is -1 raises
    KL_FLAG_BAD_PAGE; neither row is written, the valid sequence's row is."""
    x = tiny(B=3, Hq=16, Hkv=4, D=128, P=16, lens=(40, 90, 130), seed=100)
    codes, scales = fp8_cache(x)
    B, Hq, D = x["q"].shape
    v_new = torch.randn(B, 4, D, generator=torch.Generator().manual_seed(101)).to(torch.bfloat16)
    positions = torch.tensor([39, -3, 129], dtype=torch.int32)
    bt = x["block_table"].clone()
    bt[2, 129 // 16] = -1                                  # page of sequence 2's new row
    x["block_table"] = bt
    g = to_dev(x)
    sh = shape_of(x)
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, 1)), dtype=torch.uint8,
                     device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    c, s = torch.from_numpy(codes).to(_gpu.dev()), torch.from_numpy(scales).to(_gpu.dev())
    out = torch.empty(B, Hq, D, dtype=torch.float32, device=_gpu.dev())
    kl.kl_decode_step_fp8(sh, g["q"], g["w_r"], v_new.to(_gpu.dev()), positions.to(_gpu.dev()), c, s,
                          g["block_table"], g["seq_lens"], 1, out, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    flags = int(err.item())
    assert flags & kl.KL_FLAG_BAD_POSITION and flags & kl.KL_FLAG_BAD_PAGE
    want_c, want_s = oracle.append_fp8(codes, scales, bf16_bits(v_new)[:1], bt.numpy()[:1],
                                       positions.numpy()[:1])
    assert np.array_equal(c.cpu().numpy(), want_c)
    assert np.array_equal(s.cpu().numpy().view(np.uint32), want_s.view(np.uint32))
