"""Host-side pieces of bench.py on CPU (no GPU): the one-core oracle timing in a spawned process,
and the split of the oracle's sample into the pages its sequences use."""
from __future__ import annotations

import importlib.util
import os
import sys

import numpy as np

import oracle
from paper_2606_21848_gb300.workloads import bf16_bits
from tests._inputs import tiny

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    """bench.py as the module `bench` (registered, so that a spawned child finds its functions)."""
    if "bench" in sys.modules:
        return sys.modules["bench"]
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    sys.modules["bench"] = mod
    spec.loader.exec_module(mod)
    return mod


def test_one_core_oracle_runs_single_threaded_on_whole_sequences():
    x = tiny(B=6, Hq=8, Hkv=2, D=64, P=16, lens=(40, 300, 7, 129, 64, 1), seed=120)
    rate, seqs, el, cores = _bench().cpu_oracle_one_core(x, 0.5, False, max_seqs=4)
    assert cores == 1
    assert seqs >= 1 and el >= 0.5 and rate > 0


def test_one_core_sample_holds_exactly_its_sequences_pages():
    """The child decodes the first sequences from a compact pool of their own pages; the oracle
    on that pool equals the oracle on the full cache for those sequences."""
    x = tiny(B=5, Hq=8, Hkv=2, D=64, P=16, lens=(33, 200, 16, 90, 400), seed=121)
    n = 3
    q, w, v, bt, sl = _bench().oracle_sample(x, n)
    pages = sum(-(-int(L) // 16) for L in x["seq_lens"].numpy()[:n])
    assert v.shape[0] == pages < x["v_cache"].shape[0]
    full = oracle.decode(bf16_bits(x["q"])[:n], bf16_bits(x["w_r"]), bf16_bits(x["v_cache"]),
                         x["block_table"].numpy()[:n], x["seq_lens"].numpy()[:n], scale=0.125)
    assert np.array_equal(oracle.decode(q, w, v, bt, sl, scale=0.125), full)
