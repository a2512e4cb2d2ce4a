"""Helpers of the GPU parity tests: run the C-ABI path on seeded inputs, compare with the
oracle at the tolerance of the decode (bf16 inputs, fp32 accumulation)."""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300.workloads import bf16_bits

ATOL, RTOL = 2e-3, 1e-2          # |gpu - oracle| <= 2e-3 + 1e-2 |oracle|, elementwise

KERNELS = {"simt": kl.KL_KERNEL_SIMT, "tensor": kl.KL_KERNEL_TENSOR}


def dev():
    return torch.device("cuda:0")


def shape_of(x: dict, scale: float = 0.0) -> kl.kl_shape:
    wl = x["workload"]
    B, Hq, D = x["q"].shape
    num_pages, Hkv, P, _ = x["v_cache"].shape
    return kl.make_shape(B, Hq, Hkv, D, P, num_pages, x["block_table"].shape[1],
                         wl.wr_per_query_head if wl is not None else False, scale)


def to_dev(x: dict) -> dict:
    return {k: (v.to(dev()) if torch.is_tensor(v) else v) for k, v in x.items()}


def decode(g: dict, sh, *, kernel=kl.KL_KERNEL_AUTO, num_splits=0, out_dtype=kl.KL_FP32,
           k_cache=None):
    """Run keyless decode (or the K+V comparison when k_cache is given) on device inputs."""
    B, Hq, D = g["q"].shape
    dt = torch.float32 if out_dtype == kl.KL_FP32 else torch.bfloat16
    out = torch.full((B, Hq, D), float("nan"), dtype=dt, device=dev())
    err = torch.zeros(1, dtype=torch.int32, device=dev())
    nbytes = kl.kl_decode_workspace_size(sh, num_splits)
    ws = torch.zeros(max(nbytes, 256), dtype=torch.uint8, device=dev())
    opts = kl.decode_options(num_splits, kernel)
    if k_cache is None:
        kl.kl_decode_attention_ex(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                                  g["seq_lens"], opts, out, out_dtype, ws, err)
    else:
        kl.kl_standard_decode(sh, g["q"], k_cache, g["v_cache"], g["block_table"], g["seq_lens"],
                              opts, out, out_dtype, ws, err)
    torch.cuda.synchronize()
    return out, int(err.item())


def oracle_decode(x: dict, scale: float, heads=None):
    wl = x["workload"]
    return oracle.decode(bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"]),
                         x["block_table"].numpy(), x["seq_lens"].numpy(), scale=scale,
                         wr_per_query_head=bool(wl.wr_per_query_head) if wl else False,
                         heads=heads)


def default_scale(x: dict) -> float:
    return 1.0 / math.sqrt(x["q"].shape[-1])


def assert_parity(got: np.ndarray, want: np.ndarray, what: str = ""):
    got = np.asarray(got, np.float64)
    err = np.abs(got - want)
    bad = ~(err <= ATOL + RTOL * np.abs(want))      # NaN counts as bad
    assert not bad.any(), (f"{what}: {int(bad.sum())}/{bad.size} outside tolerance; "
                           f"max err {np.nanmax(err):.3e}; first at {np.argwhere(bad)[0]}")
    return float(err.max()) if err.size else 0.0
