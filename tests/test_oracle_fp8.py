"""Pins of the FP8 value-cache oracle (E4M3 codes, one fp32 scale per cached row), CPU only.

The E4M3 format is pinned against torch's float8_e4m3fn (an independent implementation of the
same OCP format); the per-row quantization against its error bound; the FP8 decode against the
bf16 decode on rows that FP8 represents exactly, and against a dense NumPy evaluation over the
dequantized rows."""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
from oracle import dense
from paper_2606_21848_gb300.workloads import bf16_bits
from tests._inputs import default_scale, tiny


def torch_e4m3_values(codes: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(codes.astype(np.uint8)).view(torch.float8_e4m3fn)
    return t.float().numpy().astype(np.float64)


def test_every_code_decodes_like_torch_float8_e4m3fn():
    codes = np.arange(256, dtype=np.uint8)
    got, want = oracle.e4m3_value(codes), torch_e4m3_values(codes)
    assert np.array_equal(np.isnan(got), np.isnan(want))
    ok = ~np.isnan(want)
    assert np.array_equal(got[ok], want[ok])
    assert got[0x7E] == 448.0 and got[1] == 2.0 ** -9 and np.isnan(got[0x7F])


def test_encoding_matches_torch_rounding_in_range():
    rng = np.random.default_rng(3)
    grid = oracle.e4m3_value(np.arange(127, dtype=np.uint8))
    mids = (grid[:-1] + grid[1:]) / 2                       # exact ties
    x = np.concatenate([rng.normal(0, 30, 4000), rng.normal(0, 0.01, 2000), grid, mids, -mids,
                        np.array([0.0, -0.0, 447.9, 448.0, 2.0 ** -10, 3 * 2.0 ** -11])])
    x = x[np.abs(x) <= 448.0].astype(np.float32)
    got = oracle.e4m3_from_f32(x)
    want = torch.from_numpy(x).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(got, want)


def test_encoding_saturates_and_picks_even_on_ties():
    assert oracle.e4m3_from_f32(np.float32(1000.0)) == 0x7E
    assert oracle.e4m3_from_f32(np.float32(-1000.0)) == 0xFE
    # 17 lies halfway between 16 (mantissa 000) and 18 (001): the even mantissa wins
    assert oracle.e4m3_value(oracle.e4m3_from_f32(np.float32(17.0))) == 16.0
    assert oracle.e4m3_value(oracle.e4m3_from_f32(np.float32(19.0))) == 20.0


def test_row_quantization_error_bound():
    """|v - scale * value(code)| <= scale * half the E4M3 spacing at |v| / scale (2^-4 relative
    for normals, 2^-10 for subnormals); the largest magnitude of a row maps to 448 exactly."""
    rng = np.random.default_rng(4)
    v = torch.from_numpy(np.concatenate([rng.normal(0, 1, (64, 128)),
                                         rng.normal(0, 1, (4, 128)) * 20.0,
                                         np.zeros((1, 128))])).to(torch.bfloat16)
    bits = bf16_bits(v)
    codes, scales = oracle.quantize_rows(bits)
    vf = dense.bf16_bits_to_f64(bits)
    deq = scales[:, None].astype(np.float64) * oracle.e4m3_value(codes)
    u = np.abs(vf) / np.where(scales > 0, scales, 1.0)[:, None]
    bound = scales[:, None] * np.maximum(u * 2.0 ** -4, 2.0 ** -10) * (1 + 1e-6)
    assert np.all(np.abs(deq - vf) <= bound + 1e-30)
    nz = scales > 0
    assert np.all(np.abs(oracle.e4m3_value(codes[nz])).max(axis=-1) == 448.0)
    assert scales[-1] == 0 and not codes[-1].any()


def test_fp8_decode_equals_bf16_decode_on_exact_rows():
    """Rows whose values are E4M3 values and whose scale is 1: the FP8 cache holds them
    exactly, so the FP8 decode equals the bf16 decode bit for bit."""
    x = tiny(B=3, Hq=8, Hkv=2, D=64, P=16, lens=(1, 37, 100))
    q, w, v, bt, sl = (bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"]),
                       x["block_table"].numpy(), x["seq_lens"].numpy())
    rng = np.random.default_rng(5)
    codes = rng.integers(0, 0x7E, size=v.shape, dtype=np.uint8) | \
        (rng.integers(0, 2, size=v.shape, dtype=np.uint8) << 7)
    codes[(codes & 0x7F) == 0x7F] = 0                      # no NaN codes
    vals = oracle.e4m3_value(codes)
    vb = bf16_bits(torch.from_numpy(vals.astype(np.float32)).to(torch.bfloat16))
    assert np.array_equal(dense.bf16_bits_to_f64(vb), vals)   # exact in bf16
    scales = np.ones(v.shape[:-1], np.float32)
    got = oracle.decode_fp8(q, w, codes, scales, bt, sl, scale=default_scale(64))
    want = oracle.decode(q, w, vb, bt, sl, scale=default_scale(64))
    np.testing.assert_array_equal(got, want)


def test_fp8_decode_equals_dense_over_dequantized_rows():
    x = tiny(B=2, Hq=8, Hkv=2, D=128, P=16, lens=(300, 41))
    q, w, v, bt, sl = (bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"]),
                       x["block_table"].numpy(), x["seq_lens"].numpy())
    codes, scales = oracle.quantize_rows(v)
    deq = scales[..., None].astype(np.float64) * torch_e4m3_values(codes)
    seqs = []
    for b, L in enumerate(sl):
        t = np.arange(int(L))
        seqs.append(np.transpose(deq[bt[b, t // 16], :, t % 16, :], (1, 0, 2)))
    qf, wf = dense.bf16_bits_to_f64(q), dense.bf16_bits_to_f64(w)
    want = np.zeros((2, 8, 128))
    for b in range(2):
        for h in range(8):
            V = seqs[b][h // 4]
            s = (V @ (qf[b, h] @ wf[h // 4])) / math.sqrt(128)
            a = np.exp(s - s.max())
            want[b, h] = (a / a.sum()) @ V
    got = oracle.decode_fp8(q, w, codes, scales, bt, sl, scale=1 / math.sqrt(128))
    np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-12)


def test_fp8_append_quantizes_the_row_in_place():
    x = tiny(B=2, Hq=4, Hkv=2, D=64, P=16, lens=(20, 33))
    v = bf16_bits(x["v_cache"])
    codes, scales = oracle.quantize_rows(v)
    v_new = bf16_bits(x["v_new"])
    bt, pos = x["block_table"].numpy(), x["positions"].numpy()
    c2, s2 = oracle.append_fp8(codes, scales, v_new, bt, pos)
    nc, ns = oracle.quantize_rows(v_new)
    for b in range(2):
        page, row = bt[b, pos[b] // 16], pos[b] % 16
        assert np.array_equal(c2[page, :, row], nc[b]) and np.array_equal(s2[page, :, row], ns[b])
    changed = (c2 != codes).any(axis=-1) | (s2 != scales)
    assert changed.sum() <= 2 * 2
