"""Dense, non-paged NumPy brute force of Keyless Attention decode (tiny inputs only).

TEST INFRASTRUCTURE, like the rest of ``oracle/``. It shares no code with the C oracle: it
un-pages the cache with its own indexing, then evaluates, per query head h of value group g,

    q_r = q_h W^R                         (Eq. 2 / Eq. 4, Section 2.2)
    s   = scale * V_g q_r                 (scores against the cached value rows, Section 3)
    a   = softmax(s)                      (alpha_{n+1,i}, Section 3)
    o   = a V_g                           (O_{n+1} = sum_i alpha_{n+1,i} v_i, Section 3)

with NumPy matrix products in fp64.
"""
from __future__ import annotations

import numpy as np


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    bits = np.asarray(bits, dtype=np.uint16)
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def unpage(v_cache_bits: np.ndarray, block_table: np.ndarray, seq_lens: np.ndarray):
    """List over sequences of dense [Hkv, L_b, D] fp64 arrays gathered from the paged cache."""
    cache = bf16_bits_to_f64(v_cache_bits)          # [num_pages, Hkv, P, D]
    P = cache.shape[2]
    seqs = []
    for b, L in enumerate(np.asarray(seq_lens)):
        t = np.arange(int(L))
        pages = np.asarray(block_table)[b, t // P]
        rows = cache[pages, :, t % P, :]            # [L, Hkv, D]
        seqs.append(np.transpose(rows, (1, 0, 2)))  # [Hkv, L, D]
    return seqs


def keyless_decode(q_bits, w_r_bits, v_seqs, *, scale: float, wr_per_query_head: bool = False):
    """Keyless decode over dense value sequences; returns [B, Hq, D] fp64."""
    q = bf16_bits_to_f64(q_bits)
    w = bf16_bits_to_f64(w_r_bits)
    B, Hq, D = q.shape
    Hkv = v_seqs[0].shape[0] if v_seqs else 1
    G = Hq // Hkv
    out = np.zeros((B, Hq, D))
    for b in range(B):
        for h in range(Hq):
            V = v_seqs[b][h // G]                    # [L, D]
            if V.shape[0] == 0:
                continue
            qr = q[b, h] @ w[h if wr_per_query_head else h // G]
            s = scale * (V @ qr)
            a = np.exp(s - s.max())
            a /= a.sum()
            out[b, h] = a @ V
    return out


def standard_decode(q_bits, k_seqs, v_seqs, *, scale: float):
    """softmax(q K^T * scale) V over dense K and V sequences (Eq. 1); [B, Hq, D] fp64."""
    q = bf16_bits_to_f64(q_bits)
    B, Hq, D = q.shape
    Hkv = v_seqs[0].shape[0] if v_seqs else 1
    G = Hq // Hkv
    out = np.zeros((B, Hq, D))
    for b in range(B):
        for h in range(Hq):
            K, V = k_seqs[b][h // G], v_seqs[b][h // G]
            if V.shape[0] == 0:
                continue
            s = scale * (K @ q[b, h])
            a = np.exp(s - s.max())
            a /= a.sum()
            out[b, h] = a @ V
    return out


def keyless_prefill(q_bits, w_r_bits, v_seqs, q_lens, *, scale: float,
                    wr_per_query_head: bool = False):
    """Keyless prefill over dense value sequences with an explicit causal mask matrix.

    Sequence b has n_b = q_lens[b] query rows (stacked in q_bits, [T, Hq, D]) for its last n_b
    positions; row i may see tokens t <= L_b - n_b + i. Returns [T, Hq, D] fp64.
    """
    q = bf16_bits_to_f64(q_bits)
    w = bf16_bits_to_f64(w_r_bits)
    T, Hq, D = q.shape
    Hkv = v_seqs[0].shape[0] if v_seqs else 1
    G = Hq // Hkv
    out = np.zeros((T, Hq, D))
    r0 = 0
    for b, n in enumerate(q_lens):
        n = int(n)
        L = v_seqs[b].shape[1]
        allowed = np.arange(L)[None, :] <= (L - n + np.arange(n))[:, None]   # [n, L]
        for h in range(Hq):
            V = v_seqs[b][h // G]                                          # [L, D]
            Qr = q[r0:r0 + n, h] @ w[h if wr_per_query_head else h // G]   # [n, D]
            s = np.where(allowed, scale * (Qr @ V.T), -np.inf)
            a = np.exp(s - s.max(axis=1, keepdims=True))
            a /= a.sum(axis=1, keepdims=True)
            out[r0:r0 + n, h] = a @ V
        r0 += n
    return out


def keyless_latent_decode(q_bits, w_r_bits, w_post_bits, lat_seqs, *, scale: float,
                          wr_per_query_head: bool = False):
    """Latent value-only cache decode by expanding the values: head h attends the rows
    V_h = V* W_post[h] (L x D) with its routed query q_r = q W^R, i.e.
    softmax(scale V_h q_r) V_h. (The oracle instead absorbs W_post into the query and expands
    only the output; the two agree by associativity.) lat_seqs from ``unpage``; [B, Hq, D]."""
    q = bf16_bits_to_f64(q_bits)
    w = bf16_bits_to_f64(w_r_bits)
    wp = bf16_bits_to_f64(w_post_bits)              # [Hq, r, D]
    B, Hq, D = q.shape
    Hl = lat_seqs[0].shape[0] if lat_seqs else 1
    G = Hq // Hl
    out = np.zeros((B, Hq, D))
    for b in range(B):
        for h in range(Hq):
            Vs = lat_seqs[b][h // G]                # [L, r]
            if Vs.shape[0] == 0:
                continue
            Vh = Vs @ wp[h]                         # [L, D]
            qr = q[b, h] @ w[h if wr_per_query_head else h // G]
            s = scale * (Vh @ qr)
            a = np.exp(s - s.max())
            a /= a.sum()
            out[b, h] = a @ Vh
    return out
