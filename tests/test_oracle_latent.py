"""Pins of the fp64 latent value-only cache decode (Section 3, latent value-only cache
paragraph), CPU only. The oracle absorbs W_post into the query and expands the output; every
expected value below comes from another association of the same product, a closed form, or a
special case that reduces to the plain keyless decode."""
from __future__ import annotations

import math

import numpy as np
import pytest

import oracle
from oracle import dense
from paper_2606_21848_gb300.workloads import bf16_bits
from tests._inputs import tiny_latent, to_bf16_bits

RTOL, ATOL = 1e-10, 1e-12


def lat_bits(x):
    return (bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["w_post"]), bf16_bits(x["v_lat"]),
            x["block_table"].numpy(), x["seq_lens"].numpy())


@pytest.mark.parametrize("shape", [
    dict(B=3, Hq=8, Hl=2, D=128, r=64, P=16, lens=(1, 37, 100)),       # group latents, r < D
    dict(B=2, Hq=8, Hl=1, D=64, r=128, P=16, lens=(70, 5)),            # one shared latent
    dict(B=2, Hq=4, Hl=4, D=64, r=32, P=8, lens=(40, 0)),              # per-head, empty sequence
])
def test_absorbed_query_equals_expanded_values(shape):
    """softmax(q* V*^T) V* W_post with q* = q_r W_post^T equals attention over the expanded
    values V* W_post (the reason only V* needs caching)."""
    x = tiny_latent(**shape)
    q, w, wp, v, bt, sl = lat_bits(x)
    scale = 1.0 / math.sqrt(shape["r"])
    got = oracle.latent_decode(q, w, wp, v, bt, sl, scale=scale)
    want = dense.keyless_latent_decode(q, w, wp, dense.unpage(v, bt, sl), scale=scale)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=ATOL)


def test_per_query_head_routing_equals_expanded_values():
    x = tiny_latent(wr_per_query_head=True)
    q, w, wp, v, bt, sl = lat_bits(x)
    got = oracle.latent_decode(q, w, wp, v, bt, sl, scale=0.1, wr_per_query_head=True)
    want = dense.keyless_latent_decode(q, w, wp, dense.unpage(v, bt, sl), scale=0.1,
                                       wr_per_query_head=True)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=ATOL)


def test_identity_expansion_is_the_plain_keyless_decode():
    """r = D and W_post = I: the latent cache is a value cache and the result is the keyless
    decode of Section 3, bit for bit."""
    x = tiny_latent(B=3, Hq=8, Hl=2, D=64, r=64, lens=(1, 37, 100))
    q, w, _, v, bt, sl = lat_bits(x)
    eye = np.broadcast_to(to_bf16_bits(np.eye(64))[None], (8, 64, 64)).copy()
    got = oracle.latent_decode(q, w, eye, v, bt, sl, scale=0.125)
    want = oracle.decode(q, w, v, bt, sl, scale=0.125)
    np.testing.assert_array_equal(got, want)


def test_single_token_returns_its_expanded_row():
    """One cached row: alpha = 1, so out = v*_0 W_post[h]."""
    x = tiny_latent(B=2, Hq=8, Hl=2, D=128, r=64, lens=(1, 1))
    q, w, wp, v, bt, sl = lat_bits(x)
    got = oracle.latent_decode(q, w, wp, v, bt, sl, scale=0.125)
    rows = dense.unpage(v, bt, sl)
    wpf = dense.bf16_bits_to_f64(wp)
    for b in range(2):
        for h in range(8):
            np.testing.assert_allclose(got[b, h], rows[b][h // 4][0] @ wpf[h], rtol=1e-12,
                                       atol=1e-13)


def test_selected_heads_match_full():
    x = tiny_latent()
    q, w, wp, v, bt, sl = lat_bits(x)
    full = oracle.latent_decode(q, w, wp, v, bt, sl, scale=0.125)
    sel = [(0, 3), (2, 7), (1, 0)]
    got = oracle.latent_decode(q, w, wp, v, bt, sl, scale=0.125, heads=sel)
    for k, (b, h) in enumerate(sel):
        np.testing.assert_array_equal(got[k], full[b, h])
