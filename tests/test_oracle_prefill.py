"""Pins of the fp64 prefill oracle (Eq. 3 under the causal mask), CPU only.

The chunked prefill is the step before decode: a chunk of n new tokens of a sequence, whose
value rows are already in the cache, attends the cached prefix and, causally, itself. Every
expected value below comes from an independent routine (the dense NumPy brute force with an
explicit mask matrix, torch SDPA in fp64), a special case of the definition, or an identity.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from oracle import dense
from tests._inputs import bits, default_scale, prefill_bits, tiny_prefill

RTOL, ATOL = 1e-10, 1e-12


@pytest.mark.parametrize("shape", [
    dict(B=3, Hq=8, Hkv=2, D=64, P=16, lens=(5, 37, 100), q_lens=(5, 12, 1)),
    dict(B=2, Hq=4, Hkv=4, D=64, P=8, lens=(33, 64), q_lens=(33, 20)),        # MHA, full + chunk
    dict(B=2, Hq=6, Hkv=1, D=32, P=16, lens=(9, 40), q_lens=(0, 17)),         # MQA, empty chunk
])
def test_paged_prefill_equals_dense_causal_bruteforce(shape):
    """Paged C oracle == dense NumPy brute force with an explicit causal mask matrix."""
    x = tiny_prefill(**shape)
    q, w, v, bt, sl, cu = prefill_bits(x)
    scale = default_scale(shape["D"])
    got = oracle.prefill(q, w, v, bt, sl, cu, scale=scale)
    want = dense.keyless_prefill(q, w, dense.unpage(v, bt, sl), shape["q_lens"], scale=scale)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=ATOL)


def test_prefill_per_query_head_routing_equals_dense():
    x = tiny_prefill(wr_per_query_head=True)
    q, w, v, bt, sl, cu = prefill_bits(x)
    assert w.shape[0] == 8
    got = oracle.prefill(q, w, v, bt, sl, cu, scale=0.1, wr_per_query_head=True)
    want = dense.keyless_prefill(q, w, dense.unpage(v, bt, sl), (5, 12, 1), scale=0.1,
                                 wr_per_query_head=True)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=ATOL)


def test_full_causal_prefill_equals_sdpa_with_k_equal_v_wr_transposed():
    """Theorem 1 (Eq. 9) with the causal mask: keyless prefill of whole sequences equals
    torch SDPA (is_causal) in fp64 with K = V (W^R)^T, an independent routine."""
    x = tiny_prefill(B=2, lens=(48, 70), q_lens=(48, 70))
    q, w, v, bt, sl, cu = prefill_bits(x)
    scale = default_scale(64)
    out = oracle.prefill(q, w, v, bt, sl, cu, scale=scale)
    qf, wf = dense.bf16_bits_to_f64(q), dense.bf16_bits_to_f64(w)
    rows = dense.unpage(v, bt, sl)
    for b in range(2):
        r0, r1 = int(cu[b]), int(cu[b + 1])
        for h in range(8):
            V = torch.from_numpy(rows[b][h // 4])
            K = V @ torch.from_numpy(wf[h // 4]).T
            Q = torch.from_numpy(qf[r0:r1, h])
            want = torch.nn.functional.scaled_dot_product_attention(
                Q[None], K[None], V[None], is_causal=True, scale=scale)[0].numpy()
            np.testing.assert_allclose(out[r0:r1, h], want, rtol=1e-10, atol=1e-12)


def test_chunk_rows_equal_decode_at_their_positions():
    """Row i of a chunk is the decode step of a sequence cut after position L - n + i: the
    decode oracle over the prefix of length L - n + i + 1 with that row as the query."""
    x = tiny_prefill(lens=(5, 37, 100), q_lens=(5, 12, 3))
    q, w, v, bt, sl, cu = prefill_bits(x)
    scale = default_scale(64)
    out = oracle.prefill(q, w, v, bt, sl, cu, scale=scale)
    for b in range(3):
        n = int(cu[b + 1] - cu[b])
        for i in range(n):
            r = int(cu[b]) + i
            L_i = int(sl[b]) - n + i + 1
            one = oracle.decode(q[r][None], w, v, bt[b][None], np.array([L_i], np.int32),
                                scale=scale)
            np.testing.assert_array_equal(out[r], one[0])


def test_first_position_returns_its_row_exactly():
    """The query at position 0 sees only token 0: alpha = 1, output = v_0 exactly."""
    x = tiny_prefill(B=2, lens=(16, 30), q_lens=(16, 30))
    q, w, v, bt, sl, cu = prefill_bits(x)
    out = oracle.prefill(q, w, v, bt, sl, cu, scale=default_scale(64))
    rows = dense.unpage(v, bt, sl)
    for b in range(2):
        for h in range(8):
            np.testing.assert_array_equal(out[int(cu[b]), h], rows[b][h // 4][0])


def test_chunked_prefill_equals_tail_of_full_prefill():
    """Splitting a sequence's prefill into a cached prefix and a chunk leaves the chunk rows
    unchanged: the last n rows of the full prefill equal the prefill of the last n rows."""
    full = tiny_prefill(B=1, lens=(90,), q_lens=(90,))
    q, w, v, bt, sl, cu = prefill_bits(full)
    scale = default_scale(64)
    whole = oracle.prefill(q, w, v, bt, sl, cu, scale=scale)
    n = 23
    tail = oracle.prefill(np.ascontiguousarray(q[90 - n:]), w, v, bt, sl,
                          np.array([0, n], np.int32), scale=scale)
    np.testing.assert_array_equal(tail, whole[90 - n:])


def test_selected_rows_match_full_prefill():
    x = tiny_prefill()
    q, w, v, bt, sl, cu = prefill_bits(x)
    full = oracle.prefill(q, w, v, bt, sl, cu, scale=0.2)
    sel = [(0, 0), (4, 7), (17, 3), (16, 1)]
    got = oracle.prefill(q, w, v, bt, sl, cu, scale=0.2, rows=sel)
    for k, (r, h) in enumerate(sel):
        np.testing.assert_array_equal(got[k], full[r, h])


def test_append_chunk_places_rows_at_the_tail():
    """Chunk rows go to positions L - n .. L - 1 of their sequence (bit copies)."""
    x = tiny_prefill(lens=(5, 37, 100), q_lens=(5, 12, 1))
    _, _, v, bt, sl, cu = prefill_bits(x)
    T, Hkv, D, P = int(cu[-1]), v.shape[1], v.shape[3], v.shape[2]
    rng = np.random.default_rng(5)
    v_new = rng.integers(0, 2**16, size=(T, Hkv, D), dtype=np.uint16)
    got = oracle.append_chunk(v, v_new, bt, sl, cu)
    want = v.copy()
    for b in range(3):
        n = int(cu[b + 1] - cu[b])
        for i in range(n):
            p = int(sl[b]) - n + i
            want[bt[b, p // P], :, p % P, :] = v_new[int(cu[b]) + i]
    np.testing.assert_array_equal(got, want)


def test_prefill_rejects_bad_offsets():
    x = tiny_prefill()
    q, w, v, bt, sl, cu = prefill_bits(x)
    with pytest.raises(ValueError):
        oracle.prefill(q, w, v, bt, sl, np.array([0, 5, 100, int(cu[-1])], np.int32), scale=0.1)
