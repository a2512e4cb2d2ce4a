"""Seeded synthetic inputs shaped like the paper's decode workloads.

This module holds random draws, page allocation and bf16 rounding only -- none of the
method's arithmetic -- so that the CUDA path and the CPU oracle can be fed the very same
bits. Everything is generated on the host with ``torch.Generator`` seeds and is returned as
CPU tensors (bf16 for q, W^R and values; int32 for tables).

Recipe (fixed, so that a seed names one input set):

1. sequence lengths: a constant, or ``randint(lo, hi + 1)`` per sequence (ragged batches);
2. q ~ N(0, 1) of shape [B, Hq, D];
3. W^R ~ N(0, wr_std^2) of shape [Hw, D, D], Hw = Hkv (one matrix per value head) or Hq;
4. the value pool [num_pages, Hkv, P, D] ~ N(0, 1), drawn in chunks of 2^24 values, chunk c
   from its own generator seeded ``seed * 1_000_003 + 7919 * (c + 1)``; with outliers, a
   Bernoulli(outlier_frac) mask per value (chunk generator seeded one higher) multiplies the
   selected fp32 values by ``outlier_scale`` before the single rounding to bf16;
5. page assignment: ``identity`` maps logical page j of sequence b to pool page
   offset_b + j; ``permuted`` applies one ``randperm(num_pages)`` to that list, which scatters
   every sequence over one shared pool. The pool holds exactly the pages the sequences use;
   block-table entries past a sequence's last page are -1;
6. the current token: ``positions = seq_lens - 1`` and v_new ~ N(0, 1) of shape [B, Hkv, D];
7. prefill workloads only (q_len > 0): the chunk of each sequence is its last
   n_b = min(q_len, L_b) rows; its queries q_chunk ~ N(0, 1) [T, Hq, D] (T = sum n_b, rows of
   sequence b at cu_q[b] ..) and its value rows v_chunk ~ N(0, 1) [T, Hkv, D] (for the chunk
   append; the pool already holds values at those rows);
8. latent workloads only (latent_dim > 0): the value pool is the latent cache (num_kv_heads =
   latent groups, head_dim = latent width = 128), and W_post ~ N(0, 1/r) of shape [Hq, r, D]
   is drawn last.
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, replace

import torch

_CHUNK = 1 << 24


@dataclass(frozen=True)
class Workload:
    name: str
    num_seqs: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    page_size: int
    seq_len: int = 0                      # uniform length (tokens, incl. the current one)
    seq_len_range: tuple[int, int] | None = None   # ragged: uniform integer in [lo, hi]
    table: str = "permuted"               # "identity" or "permuted"
    wr_std: float = 1.0
    outlier_frac: float = 0.0
    outlier_scale: float = 1.0
    wr_per_query_head: bool = False
    num_splits: int = 0                   # 0: the library chooses
    seed: int = 0
    q_len: int = 0                        # prefill: query rows per sequence (its last rows)
    latent_dim: int = 0                   # latent cache: r (the pool holds the latent rows)

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def max_seq_len(self) -> int:
        return self.seq_len_range[1] if self.seq_len_range else self.seq_len

    @property
    def max_pages_per_seq(self) -> int:
        return max(1, math.ceil(self.max_seq_len / self.page_size))

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


# The five decode workloads: Qwen2/Llama-style GQA shapes (head dim 64/128, groups of 4 and 8)
# as in the paper's inference-efficiency study and architecture tables.
WORKLOADS: dict[str, Workload] = {
    "tiny_mha": Workload("tiny_mha", 1, 4, 4, 64, 16, seq_len=256, table="identity",
                         wr_std=math.sqrt(1 / 64), seed=0),
    "small_gqa": Workload("small_gqa", 8, 32, 8, 128, 16, seq_len=4096,
                          wr_std=math.sqrt(1 / 128), seed=1),
    "long_context": Workload("long_context", 1, 32, 8, 128, 16, seq_len=131072,
                             wr_std=math.sqrt(1 / 128), num_splits=128, seed=2),
    "ragged_serving": Workload("ragged_serving", 64, 32, 8, 128, 16,
                               seq_len_range=(512, 32768), wr_std=math.sqrt(1 / 128),
                               outlier_frac=0.01, outlier_scale=20.0, seed=3),
    "high_concurrency_70b": Workload("high_concurrency_70b", 256, 64, 8, 128, 32, seq_len=8192,
                                     wr_std=math.sqrt(1 / 128), seed=4),
}

ORDER = ["tiny_mha", "small_gqa", "long_context", "ragged_serving", "high_concurrency_70b"]

# Groups of more than 8 query heads per value head (Section 3, multi-query and grouped-query
# attention): all 32 heads of a sequence on one value head (MQA), and 128 query heads over 8
# value heads (groups of 16).
WORKLOADS.update({
    "mqa_group32": Workload("mqa_group32", 256, 32, 1, 128, 16, seq_len=8192,
                            wr_std=math.sqrt(1 / 128), seed=8),
    "gqa_group16": Workload("gqa_group16", 64, 128, 8, 128, 32, seq_len=8192,
                            wr_std=math.sqrt(1 / 128), seed=9),
})
LARGE_GROUPS = ["mqa_group32", "gqa_group16"]

# Head dim 64 (GPT-2's head layout, the paper's main experiments): 16 heads of 64 dims, multi-head
# (one value head per query head), batch 32 at 8192 tokens -- 512 MiB of cached values.
WORKLOADS.update({
    "mha_d64": Workload("mha_d64", 32, 16, 16, 64, 16, seq_len=8192, wr_std=math.sqrt(1 / 64),
                        seed=10),
})
EXTRA = LARGE_GROUPS + ["mha_d64"]

# Prefill workloads (chunked prefill, the step before decode): a whole 32K-token prompt with
# the paper's Qwen2-1.5B attention (12 query heads, 2 value heads, head dim 128, W^R per query
# head, trained at 32,768 tokens), and a serving-style chunk of 512 new tokens on an
# 8192-token sequence (7680 cached) for a batch of 8, GQA 32 / 8.
WORKLOADS.update({
    "prefill_qwen2_32k": Workload("prefill_qwen2_32k", 1, 12, 2, 128, 16, seq_len=32768,
                                  wr_std=math.sqrt(1 / 128), wr_per_query_head=True, seed=5,
                                  q_len=32768),
    "prefill_chunked_gqa": Workload("prefill_chunked_gqa", 8, 32, 8, 128, 16, seq_len=8192,
                                    wr_std=math.sqrt(1 / 128), seed=6, q_len=512),
})

# Latent value-only cache workload (Section 3): 32 query heads reading 4 latent groups of width
# 128 (8 heads per group), batch 64 at 8192 tokens, W_post per query head: 1 KiB of cache per
# token, half of a 8-value-head value-only cache and a quarter of its K+V cache.
WORKLOADS.update({
    "latent_serving": Workload("latent_serving", 64, 32, 4, 128, 16, seq_len=8192,
                               wr_std=math.sqrt(1 / 128), seed=7, latent_dim=128),
})


def _pool_chunk(args):
    out_flat, c, n, seed, frac, scale = args
    g = torch.Generator().manual_seed(seed * 1_000_003 + 7919 * (c + 1))
    x = torch.randn(n, generator=g)
    if frac > 0.0:
        gm = torch.Generator().manual_seed(seed * 1_000_003 + 7919 * (c + 1) + 1)
        mask = torch.rand(n, generator=gm) < frac
        x = torch.where(mask, x * scale, x)
    out_flat[c * _CHUNK: c * _CHUNK + n].copy_(x)


def value_pool(num_values: int, seed: int, frac: float = 0.0, scale: float = 1.0,
               threads: int | None = None) -> torch.Tensor:
    """Flat bf16 tensor of N(0,1) values (with optional outliers), chunked as in the recipe."""
    out = torch.empty(num_values, dtype=torch.bfloat16)
    n_chunks = (num_values + _CHUNK - 1) // _CHUNK
    jobs = [(out, c, min(_CHUNK, num_values - c * _CHUNK), seed, frac, scale)
            for c in range(n_chunks)]
    threads = threads or min(16, os.cpu_count() or 1)
    if n_chunks == 1 or threads == 1:
        for j in jobs:
            _pool_chunk(j)
    else:
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(_pool_chunk, jobs))
    return out


def generate(wl: Workload, seed: int | None = None) -> dict:
    """Inputs of one decode step of workload `wl` as CPU tensors (see the module recipe)."""
    seed = wl.seed if seed is None else seed
    g = torch.Generator().manual_seed(seed)
    B, Hq, Hkv, D, P = wl.num_seqs, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.page_size

    if wl.seq_len_range is not None:
        lo, hi = wl.seq_len_range
        seq_lens = torch.randint(lo, hi + 1, (B,), generator=g, dtype=torch.int64)
    else:
        seq_lens = torch.full((B,), wl.seq_len, dtype=torch.int64)
    seq_lens = seq_lens.to(torch.int32)

    q = torch.randn(B, Hq, D, generator=g).to(torch.bfloat16)
    Hw = Hq if wl.wr_per_query_head else Hkv
    w_r = (torch.randn(Hw, D, D, generator=g) * wl.wr_std).to(torch.bfloat16)

    pages_per_seq = [max(0, math.ceil(int(L) / P)) for L in seq_lens.tolist()]
    num_pages = max(1, sum(pages_per_seq))
    v_cache = value_pool(num_pages * Hkv * P * D, seed, wl.outlier_frac,
                         wl.outlier_scale).view(num_pages, Hkv, P, D)

    if wl.table == "identity":
        pool_ids = torch.arange(num_pages, dtype=torch.int64)
    else:
        pool_ids = torch.randperm(num_pages, generator=g)
    max_pages = wl.max_pages_per_seq
    block_table = torch.full((B, max_pages), -1, dtype=torch.int32)
    off = 0
    for b, n in enumerate(pages_per_seq):
        block_table[b, :n] = pool_ids[off: off + n].to(torch.int32)
        off += n

    positions = (seq_lens - 1).clamp_min(0).to(torch.int32)
    v_new = torch.randn(B, Hkv, D, generator=g).to(torch.bfloat16)
    out = dict(q=q, w_r=w_r, v_cache=v_cache, block_table=block_table, seq_lens=seq_lens,
               positions=positions, v_new=v_new, num_pages=num_pages, workload=wl)
    if wl.q_len > 0:
        q_lens = torch.clamp(seq_lens, max=wl.q_len).to(torch.int32)
        cu_q = torch.zeros(B + 1, dtype=torch.int32)
        cu_q[1:] = torch.cumsum(q_lens, 0).to(torch.int32)
        T = int(cu_q[-1])
        out.update(q_chunk=torch.randn(T, Hq, D, generator=g).to(torch.bfloat16),
                   v_chunk=torch.randn(T, Hkv, D, generator=g).to(torch.bfloat16),
                   q_lens=q_lens, cu_q=cu_q)
    if wl.latent_dim > 0:
        r = wl.latent_dim
        assert r == D, "the value pool doubles as the latent cache"
        out["w_post"] = (torch.randn(Hq, r, D, generator=g) * math.sqrt(1.0 / r)).to(torch.bfloat16)
        out["v_lat"] = v_cache
    return out


def bf16_bits(t: torch.Tensor):
    """uint16 NumPy view of a bf16 CPU tensor's bit patterns (no arithmetic)."""
    assert t.dtype == torch.bfloat16
    return t.contiguous().view(torch.int16).numpy().view("uint16")
