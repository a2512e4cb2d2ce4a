"""Pins of the fp64 oracle against what the paper and the mathematics fix (CPU only).

Each test states the passage or identity it pins. The oracle is never compared with itself:
every expected value comes from a closed form, an invariant, an independent dense routine
(NumPy or torch SDPA in fp64), or a special case of the definition.
"""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
from oracle import dense
from tests._inputs import bits, default_scale, tiny, to_bf16_bits

RTOL, ATOL = 1e-10, 1e-12


@pytest.mark.parametrize("shape", [
    dict(B=3, Hq=8, Hkv=2, D=64, P=16, lens=(1, 37, 100)),          # GQA, group 4
    dict(B=2, Hq=4, Hkv=4, D=64, P=16, lens=(256, 17)),              # MHA
    dict(B=2, Hq=6, Hkv=1, D=32, P=8, lens=(9, 40)),                 # MQA (Section 3)
    dict(B=2, Hq=8, Hkv=2, D=128, P=32, lens=(70, 0)),               # empty sequence
])
def test_paged_oracle_equals_dense_bruteforce(shape):
    """Paged C oracle == dense, non-paged NumPy brute force (Section 3 decode formula)."""
    x = tiny(**shape)
    q, w, v, bt, sl = bits(x)
    scale = default_scale(shape["D"])
    got = oracle.decode(q, w, v, bt, sl, scale=scale)
    want = dense.keyless_decode(q, w, dense.unpage(v, bt, sl), scale=scale)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=ATOL)


def test_per_query_head_routing_equals_dense():
    """W^R made head-specific (one matrix per query head, Section 5.4 / Appendix B)."""
    x = tiny(wr_per_query_head=True)
    q, w, v, bt, sl = bits(x)
    assert w.shape[0] == 8
    got = oracle.decode(q, w, v, bt, sl, scale=0.1, wr_per_query_head=True)
    want = dense.keyless_decode(q, w, dense.unpage(v, bt, sl), scale=0.1, wr_per_query_head=True)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=ATOL)


def test_softmax_weights_sum_to_one():
    """alpha_{n+1,i} is a softmax over the n+1 cached rows (Section 3): sum = 1, all > 0."""
    x = tiny(lens=(1, 200, 63))
    q, w, v, bt, sl = bits(x)
    for b in range(3):
        for h in (0, 5):
            a = oracle.attention_weights(q, w, v, bt, sl, b, h, scale=default_scale(64))
            assert a.shape == (int(sl[b]),)
            assert np.all(a > 0)
            assert abs(a.sum() - 1.0) < 1e-12


def test_single_token_returns_its_row_exactly():
    """n+1 = 1: alpha = 1, so O equals the one cached value row (Section 3)."""
    x = tiny(lens=(1, 1, 1))
    q, w, v, bt, sl = bits(x)
    out = oracle.decode(q, w, v, bt, sl, scale=default_scale(64))
    rows = dense.unpage(v, bt, sl)
    for b in range(3):
        for h in range(8):
            np.testing.assert_array_equal(out[b, h], rows[b][h // 4][0])


def test_uniform_values_give_that_value():
    """All cached rows equal u: O = u sum_i alpha_i = u for any query and W^R."""
    x = tiny(lens=(5, 64, 99))
    q, w, v, bt, sl = bits(x)
    u = np.random.default_rng(0).standard_normal((2, 64))
    ub = to_bf16_bits(u)
    v = np.broadcast_to(ub[None, :, None, :], v.shape).copy()
    out = oracle.decode(q, w, v, bt, sl, scale=default_scale(64))
    uf = dense.bf16_bits_to_f64(ub)
    for h in range(8):
        np.testing.assert_allclose(out[:, h], np.broadcast_to(uf[h // 4], (3, 64)), rtol=1e-13)


def test_group_mapping_reads_value_head_h_over_g():
    """GQA (Section 3): heads of group g share V_g. Constant V per group pins h -> h // G."""
    x = tiny(B=2, Hq=8, Hkv=4, lens=(10, 33))
    q, w, v, bt, sl = bits(x)
    consts = to_bf16_bits(np.arange(1, 5, dtype=np.float64))           # value head g -> g + 1
    v = np.broadcast_to(consts[None, :, None, None], v.shape).copy()
    out = oracle.decode(q, w, v, bt, sl, scale=default_scale(64))
    for h in range(8):
        np.testing.assert_allclose(out[:, h], h // 2 + 1.0, rtol=1e-13)


@pytest.mark.parametrize("zero", ["q", "w_r"])
def test_zero_query_or_routing_gives_mean_of_rows(zero):
    """q = 0 or W^R = 0: every score is 0, alpha = 1/(n+1), O = mean of the cached rows."""
    x = tiny(lens=(3, 50, 128))
    q, w, v, bt, sl = bits(x)
    if zero == "q":
        q = np.zeros_like(q)
    else:
        w = np.zeros_like(w)
    out = oracle.decode(q, w, v, bt, sl, scale=default_scale(64))
    rows = dense.unpage(v, bt, sl)
    for b in range(3):
        for h in range(8):
            np.testing.assert_allclose(out[b, h], rows[b][h // 4].mean(axis=0), rtol=1e-12,
                                       atol=1e-14)


def test_dominant_score_selects_that_row():
    """A routed query aligned with one row and scaled up: alpha -> one-hot, O -> that row."""
    x = tiny(B=1, Hq=2, Hkv=1, D=64, lens=(80,))
    _, _, v, bt, sl = bits(x)
    rows = dense.unpage(v, bt, sl)[0][0]
    t = 41
    w = to_bf16_bits(np.eye(64))[None]                  # W^R = I
    q = to_bf16_bits(64.0 * rows[t])[None, None].repeat(2, axis=1)  # exact: power-of-two scale
    out = oracle.decode(q, w, v, bt, sl, scale=default_scale(64))
    np.testing.assert_allclose(out[0, 0], rows[t], rtol=0, atol=1e-12)


def _sdpa_fp64(qv, K, V, scale):
    """torch scaled_dot_product_attention in fp64 for one query row."""
    return torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(qv)[None, None], torch.from_numpy(K)[None], torch.from_numpy(V)[None],
        scale=scale)[0, 0].numpy()


def test_theorem1_keyless_equals_standard_attention_with_k_equal_v_wr_transposed():
    """Theorem 1 / Eq. 9: q W^R v^T = q (v (W^R)^T)^T, so keyless attention equals standard
    attention with K = V (W^R)^T. Checked against torch SDPA in fp64 (an independent routine)."""
    x = tiny(lens=(7, 90, 128))
    q, w, v, bt, sl = bits(x)
    scale = default_scale(64)
    out = oracle.decode(q, w, v, bt, sl, scale=scale)
    qf, wf = dense.bf16_bits_to_f64(q), dense.bf16_bits_to_f64(w)
    rows = dense.unpage(v, bt, sl)
    for b in range(3):
        for h in range(8):
            V = rows[b][h // 4]
            K = V @ wf[h // 4].T
            np.testing.assert_allclose(out[b, h], _sdpa_fp64(qf[b, h], K, V, scale),
                                       rtol=1e-10, atol=1e-12)


def test_identity_routing_is_kv_sharing():
    """W^R = I is QVV(2), the KV-sharing method (Section 5.3): scores q . v / sqrt(d_k)."""
    x = tiny(lens=(12, 77, 3))
    q, _, v, bt, sl = bits(x)
    w = np.broadcast_to(to_bf16_bits(np.eye(64))[None], (2, 64, 64)).copy()
    out = oracle.decode(q, w, v, bt, sl, scale=default_scale(64))
    qf = dense.bf16_bits_to_f64(q)
    rows = dense.unpage(v, bt, sl)
    for b in range(3):
        for h in range(8):
            V = rows[b][h // 4]
            np.testing.assert_allclose(out[b, h], _sdpa_fp64(qf[b, h], V, V, default_scale(64)),
                                       rtol=1e-10, atol=1e-12)


def test_page_permutation_invariance_is_bit_exact():
    """Moving physical pages (and rewriting the block table) cannot change any result."""
    x = tiny(lens=(40, 100, 17))
    q, w, v, bt, sl = bits(x)
    out1 = oracle.decode(q, w, v, bt, sl, scale=default_scale(64))
    perm = np.random.default_rng(3).permutation(v.shape[0])   # new page p holds old perm[p]
    inv = np.argsort(perm)
    v2 = v[perm]
    bt2 = np.where(bt >= 0, inv[np.maximum(bt, 0)], -1).astype(np.int32)
    out2 = oracle.decode(q, w, v2, bt2, sl, scale=default_scale(64))
    np.testing.assert_array_equal(out1, out2)


@pytest.mark.parametrize("chunk", [1, 16, 33, 128])
def test_split_merge_identity(chunk):
    """Combining split states of any partition of [0, n+1) equals the unsplit softmax."""
    x = tiny(lens=(1, 100, 128))
    q, w, v, bt, sl = bits(x)
    S = math.ceil(128 / chunk)
    po, pml = oracle.decode_partial(q, w, v, bt, sl, scale=0.2, chunk=chunk, num_splits=S)
    merged = oracle.combine(po, pml)
    full = oracle.decode(q, w, v, bt, sl, scale=0.2)
    np.testing.assert_allclose(merged, full, rtol=1e-12, atol=1e-14)
    # empty splits are marked l = 0 and skipped
    assert np.all(pml[0, :, 1:, 1] == 0.0)


def test_combine_closed_form_two_splits():
    """Two splits with m = (0, ln 3), l = (1, 1): weights 1 : 3, so O = (o1 + 3 o2) / 4."""
    po = np.zeros((1, 1, 2, 4))
    po[0, 0, 0] = [1, 2, 3, 4]
    po[0, 0, 1] = [5, 6, 7, 8]
    pml = np.array([[[[0.0, 1.0], [math.log(3.0), 1.0]]]])
    np.testing.assert_allclose(oracle.combine(po, pml)[0, 0],
                               (po[0, 0, 0] + 3 * po[0, 0, 1]) / 4, rtol=1e-14)


def test_standard_decode_matches_dense():
    """The K+V comparison oracle (Eq. 1) against its dense NumPy counterpart."""
    x = tiny(lens=(31, 64, 1))
    q, _, v, bt, sl = bits(x)
    k = to_bf16_bits(np.random.default_rng(5).standard_normal(v.shape))
    got = oracle.standard_decode(q, k, v, bt, sl, scale=0.125)
    want = dense.standard_decode(q, dense.unpage(k, bt, sl), dense.unpage(v, bt, sl), scale=0.125)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=ATOL)


def test_route_matches_row_times_matrix():
    """q_r = q W^R with q a row vector (Section 2.2), against NumPy matmul."""
    x = tiny()
    q, w = bits(x)[:2]
    qr = oracle.route(q, w, num_kv_heads=2)
    qf, wf = dense.bf16_bits_to_f64(q), dense.bf16_bits_to_f64(w)
    for h in range(8):
        np.testing.assert_allclose(qr[:, h], qf[:, h] @ wf[h // 4], rtol=1e-12, atol=1e-14)


def test_append_places_row_at_position():
    """The current token's value row lands at row positions[b] of the sequence (Section 3)."""
    x = tiny(lens=(16, 45, 100))
    q, w, v, bt, sl = bits(x)
    vn = to_bf16_bits(np.random.default_rng(9).standard_normal((3, 2, 64)))
    pos = np.array([15, 44, 60], np.int32)
    v2 = oracle.append(v, vn, bt, pos)
    rows_before = dense.unpage(v, bt, sl)
    rows_after = dense.unpage(v2, bt, sl)
    for b in range(3):
        for g in range(2):
            np.testing.assert_array_equal(v2.view(np.uint16)[bt[b, pos[b] // 16], g, pos[b] % 16],
                                          vn[b, g])
            mask = np.ones(int(sl[b]), bool)
            mask[pos[b]] = False
            np.testing.assert_array_equal(rows_after[b][g][mask], rows_before[b][g][mask])
    # exactly B * Hkv rows changed
    assert int(np.sum(np.any(v2 != v, axis=-1))) <= 3 * 2


def test_out_of_range_page_is_rejected():
    x = tiny(lens=(20, 40, 60))
    q, w, v, bt, sl = bits(x)
    bt = bt.copy()
    bt[1, 1] = v.shape[0]
    with pytest.raises(ValueError):
        oracle.decode(q, w, v, bt, sl, scale=0.1)
