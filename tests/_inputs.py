"""Small seeded input sets shared by the oracle pins and the GPU parity tests."""
from __future__ import annotations

import math

import numpy as np
import torch

from paper_2606_21848_gb300.workloads import Workload, bf16_bits, generate


def tiny(B=3, Hq=8, Hkv=2, D=64, P=16, lens=(1, 37, 100), seed=11, table="permuted",
         wr_per_query_head=False, wr_std=None):
    """A tiny ragged workload with explicit lengths (bypasses the length draw)."""
    wl = Workload("test", B, Hq, Hkv, D, P, seq_len=max(lens), table=table,
                  wr_std=wr_std if wr_std is not None else math.sqrt(1.0 / D),
                  wr_per_query_head=wr_per_query_head, seed=seed)
    x = generate(wl)
    # Re-allocate pages for the explicit lengths so the pool holds exactly the pages used.
    g = torch.Generator().manual_seed(seed + 99)
    lens_t = torch.tensor(lens, dtype=torch.int32)
    pages = [math.ceil(L / P) for L in lens]
    num_pages = max(1, sum(pages))
    v = (torch.randn(num_pages, Hkv, P, D, generator=g)).to(torch.bfloat16)
    ids = torch.arange(num_pages) if table == "identity" else torch.randperm(num_pages, generator=g)
    bt = torch.full((B, max(1, max(pages))), -1, dtype=torch.int32)
    off = 0
    for b, n in enumerate(pages):
        bt[b, :n] = ids[off: off + n].to(torch.int32)
        off += n
    x.update(v_cache=v, block_table=bt, seq_lens=lens_t, num_pages=num_pages,
             positions=(lens_t - 1).clamp_min(0).to(torch.int32))
    return x


def bits(x: dict):
    """NumPy views for the oracle: (q, w_r, v_cache, block_table, seq_lens)."""
    return (bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"]),
            x["block_table"].numpy(), x["seq_lens"].numpy())


def default_scale(D: int) -> float:
    return 1.0 / math.sqrt(D)


def to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round fp64/fp32 values to bf16 (round-to-nearest-even, via torch) and return the bits."""
    return bf16_bits(torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16))


def tiny_prefill(B=3, Hq=8, Hkv=2, D=64, P=16, lens=(5, 37, 100), q_lens=(5, 12, 1), seed=21,
                 table="permuted", wr_per_query_head=False):
    """A tiny chunked-prefill input: the cache of ``tiny`` plus a chunk of q_lens[b] query rows
    for the last q_lens[b] positions of each sequence (q is [T, Hq, D], cu_q its row offsets)."""
    assert all(0 <= n <= L for n, L in zip(q_lens, lens))
    x = tiny(B, Hq, Hkv, D, P, lens, seed, table, wr_per_query_head)
    g = torch.Generator().manual_seed(seed + 7)
    T = int(sum(q_lens))
    x["q"] = torch.randn(T, Hq, D, generator=g).to(torch.bfloat16)
    x["cu_q"] = torch.tensor(np.concatenate([[0], np.cumsum(q_lens)]), dtype=torch.int32)
    x["q_lens"] = torch.tensor(q_lens, dtype=torch.int32)
    return x


def prefill_bits(x: dict):
    """NumPy views for the prefill oracle: (q, w_r, v_cache, block_table, seq_lens, cu_q)."""
    return bits(x) + (x["cu_q"].numpy(),)


def tiny_latent(B=3, Hq=8, Hl=2, D=128, r=64, P=16, lens=(1, 37, 100), seed=51,
                table="permuted", wr_per_query_head=False):
    """A tiny decode over a latent value-only cache: latent rows [pages][Hl][P][r] ~ N(0, 1),
    W_post [Hq][r][D] ~ N(0, 1/r) (so that the expanded values are ~ N(0, 1)), q and W^R as in
    ``tiny``."""
    x = tiny(B, Hq, Hl, D, P, lens, seed, table, wr_per_query_head)
    g = torch.Generator().manual_seed(seed + 13)
    num_pages = x["num_pages"]
    x["v_lat"] = torch.randn(num_pages, Hl, P, r, generator=g).to(torch.bfloat16)
    x["w_post"] = (torch.randn(Hq, r, D, generator=g) * math.sqrt(1.0 / r)).to(torch.bfloat16)
    x["r"] = r
    return x
