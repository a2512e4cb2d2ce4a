"""Benchmark of one keyless decode step (append + decode attention) on GB300.

A step is one pass of the whole hot path over one batch: kl_decode_step appends the current
token's value rows to the paged Value-Only Cache and runs the routed decode (routing prologue,
split-sequence decode, cross-split merge) -- one kernel on the tensor-core path (the last split
of each sequence and value head merges the split states), the decode kernel plus the combine
kernel on the CUDA-core path. Inputs are
seeded synthetic tensors with the shapes of the selected workload, resident in HBM before the
timed region; L2 is flushed between timed steps (a 512 MiB write, then a read of it, so the
lines left in L2 are clean).

Prints ONE JSON line (rank 0). `--impl reference` times the fp64 CPU oracle instead (the
reference arm: a slow CPU program, timed on a bounded sample of the same workload).
`--workload prefill_*` times the chunked prefill instead: one step = the chunk append plus the
prefill attention, reported as query tokens/s against the bf16 tensor roofline.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

# The large-batch workload: batch 256, 64/8 heads, D 128, 8192 tokens, P 32 (4 GiB of cached
# values). The metric's ">= 80% of 8 TB/s" target is stated for the long-context and
# large-batch workloads; this is the larger of the two. Others: --workload NAME.
DEFAULT_WORKLOAD = "high_concurrency_70b"
METRIC = "decode attention tokens/s and achieved HBM GB/s (% of 8 TB/s) on 1 GB300"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=50)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default=DEFAULT_WORKLOAD)
    p.add_argument("--kernel", default="auto", choices=["auto", "tensor", "simt"])
    p.add_argument("--num-splits", type=int, default=-1, help="-1: the workload's setting")
    p.add_argument("--standard", action="store_true",
                   help="time the same-design K+V decode (comparison) instead of keyless")
    p.add_argument("--wr-per-query-head", action="store_true",
                   help="one W^R per query head (the paper's GQA models) instead of per value head")
    p.add_argument("--fused-query", action="store_true",
                   help="decode with the composed query q = x W^Q W^R (no W^R in the kernel)")
    p.add_argument("--fp8-cache", action="store_true",
                   help="FP8 (E4M3, per-row scale) value cache: quantizing append + FP8 decode")
    p.add_argument("--num-seqs", type=int, default=0,
                   help="override the workload's batch size (decode workloads; 0: as defined)")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-sweep", action="store_true",
                   help="skip the other workloads (measured after the default line)")
    p.add_argument("--cpu-seconds", type=float, default=10.0)
    return p.parse_args()


# ------------------------------------------------------------------------------ helpers --

def dist_env():
    from paper_2606_21848_gb300.multi import dist_env as env
    return env()


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# the sources each decode kernel is compiled from (traffic records are keyed to their hash)
DECODE_SOURCES = ("kl_decode_tc.cu", "kl_decode_tc64.cu", "kl_decode_tc_groups.cu",
                  "kl_decode_tc_kernel.cuh",
                  "kl_internal.cuh", "kl_tc_ptx.cuh")
FP8_SOURCES = ("kl_decode_fp8.cu", "kl_fp8_quant.cuh", "kl_internal.cuh", "kl_tc_ptx.cuh")


def kernel_source_digest(names=DECODE_SOURCES) -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2606_21848_gb300", "csrc")
    for name in sorted(names):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(workload: str, kernel: str):
    """DRAM bytes per launch from the committed ncu summary, if taken on the current source."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.md")
    if not os.path.exists(path):
        return None
    digest = kernel_source_digest(FP8_SOURCES if kernel == "tensor-fp8" else DECODE_SOURCES)
    for line in open(path):
        m = re.match(r"\|\s*(\S+)\s*\|\s*(\S+)\s*\|\s*([0-9]+)\s*\|\s*([0-9a-f]+)\s*\|", line)
        if m and m.group(1) == workload and m.group(2) == kernel and m.group(4) == digest:
            return int(m.group(3))
    return None


class ClockSampler:
    """nvidia-smi clock / throttle-reason sampling while the timed region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.idx)], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
                out = ""
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        if not getattr(self, "lines", None):
            return None
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in self.lines:
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = max(mx, float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() in ("active", "1"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def algorithmic_bytes(x, standard: bool, with_wr: bool = True, fp8: bool = False) -> dict:
    """Bytes the decode must move once: cached rows (V, plus K for the comparison), W^R,
    q, out (fp32 read by nobody: bf16 written), block table and lengths."""
    wl = x["workload"]
    B, Hq, D = x["q"].shape
    Hkv = x["v_cache"].shape[1]
    P = x["v_cache"].shape[2]
    tokens = int(x["seq_lens"].sum())
    v = tokens * Hkv * (D + 4) if fp8 else tokens * Hkv * D * 2     # codes + row scale
    cache = 2 * v if standard else v
    wr = 0 if standard or not with_wr else x["w_r"].numel() * 2
    q = B * Hq * D * 2
    out = B * Hq * D * 2
    bt = sum(math.ceil(int(L) / P) for L in x["seq_lens"].tolist()) * 4 + B * 4
    # v_new read + the cache row written (bf16, or codes and scale)
    append = 0 if standard else B * Hkv * (D * 2 + (D + 4 if fp8 else D * 2))
    return {"cache": cache, "wr": wr, "total": cache + wr + q + out + bt + append,
            "tokens": tokens}


# ----------------------------------------------------------------------------- CPU arm --

def cpu_oracle_rate(x, seconds: float, standard: bool):
    """Time the fp64 oracle (as it stands) on whole sequences until `seconds` pass."""
    import numpy as np

    import oracle
    from paper_2606_21848_gb300.workloads import bf16_bits

    q, w, v = bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"])
    bt, sl = x["block_table"].numpy(), x["seq_lens"].numpy()
    B, Hq, D = x["q"].shape
    scale = 1.0 / math.sqrt(D)
    oracle.build()
    seqs = 0
    t0 = time.perf_counter()
    b = 0
    while True:
        heads = np.array([(b, h) for h in range(Hq)], np.int32)
        if standard:
            oracle.standard_decode(q, v, v, bt, sl, scale=scale, heads=heads)
        else:
            oracle.decode(q, w, v, bt, sl, scale=scale, heads=heads)
        seqs += 1
        b = (b + 1) % B
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    return seqs / el, seqs, el


def stage_inputs(x, names, dev):
    """A step's inputs staged for one host-to-device copy: one pinned host buffer and one device
    buffer with 256-byte-aligned sections, and the device views the kernels take.
    Returns (host buffer, device buffer, {name: device view})."""
    import torch

    nbytes = {k: x[k].numel() * x[k].element_size() for k in names}
    offs, total = {}, 0
    for k in names:
        offs[k] = total
        total += (nbytes[k] + 255) // 256 * 256
    h_stage = torch.empty(total, dtype=torch.uint8).pin_memory()
    d_stage = torch.empty(total, dtype=torch.uint8, device=dev)
    for k in names:
        h_stage[offs[k]:offs[k] + nbytes[k]].copy_(x[k].contiguous().view(-1).view(torch.uint8))
    d_in = {k: d_stage[offs[k]:offs[k] + nbytes[k]].view(x[k].dtype).view(x[k].shape)
            for k in names}
    return h_stage, d_stage, d_in


def _one_core_worker(sample, scale, standard, seconds, queue):
    """Child process: the oracle with one OpenMP thread over the sample's sequences."""
    import numpy as np

    import oracle

    q, w, v, bt, sl = sample
    B, Hq = q.shape[0], q.shape[1]
    seqs, t0, b = 0, time.perf_counter(), 0
    while True:
        heads = np.array([(b, h) for h in range(Hq)], np.int32)
        if standard:
            oracle.standard_decode(q, v, v, bt, sl, scale=scale, heads=heads)
        else:
            oracle.decode(q, w, v, bt, sl, scale=scale, heads=heads)
        seqs += 1
        b = (b + 1) % B
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    queue.put((oracle.threads(), seqs, el))


def oracle_sample(x, n: int):
    """The oracle's inputs (bf16 bits) for the batch's first n sequences over a compact pool of
    only their own pages: (q, w_r, v_cache, block_table, seq_lens), block table renumbered."""
    import numpy as np

    from paper_2606_21848_gb300.workloads import bf16_bits

    P = x["v_cache"].shape[2]
    bt_all, sl = x["block_table"].numpy()[:n], x["seq_lens"].numpy()[:n].copy()
    used = sorted({int(p) for b in range(n) for p in bt_all[b, :(int(sl[b]) + P - 1) // P]})
    remap = {p: i for i, p in enumerate(used)}
    bt = np.full_like(bt_all, -1)
    for b in range(n):
        for j in range((int(sl[b]) + P - 1) // P):
            bt[b, j] = remap[int(bt_all[b, j])]
    v = np.ascontiguousarray(bf16_bits(x["v_cache"])[used] if used else bf16_bits(x["v_cache"])[:1])
    return np.ascontiguousarray(bf16_bits(x["q"])[:n]), bf16_bits(x["w_r"]), v, bt, sl


def cpu_oracle_one_core(x, seconds: float, standard: bool, max_seqs: int = 4):
    """The oracle on one host core (OMP_NUM_THREADS=1) over the first `max_seqs` sequences,
    gathered with their own pages; run in a spawned process (this one holds a CUDA context, and
    the OpenMP thread count is fixed when the oracle library loads)."""
    import multiprocessing as mp

    sample = oracle_sample(x, min(max_seqs, x["q"].shape[0]))
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    old = os.environ.get("OMP_NUM_THREADS")
    os.environ["OMP_NUM_THREADS"] = "1"
    try:
        proc = ctx.Process(target=_one_core_worker,
                           args=(sample, 1.0 / math.sqrt(x["q"].shape[2]), standard, seconds, queue))
        proc.start()
    finally:
        if old is None:
            del os.environ["OMP_NUM_THREADS"]
        else:
            os.environ["OMP_NUM_THREADS"] = old
    cores, seqs, el = queue.get(timeout=seconds + 300)
    proc.join(timeout=60)
    return seqs / el, seqs, el, cores


def reference_steps(run_unit, args):
    """Time the oracle as the reference arm: `args.warmup` untimed steps, then `args.steps`
    timed steps, each a bounded sample of the workload (the same number of units -- whole
    sequences, or query rows -- handed to `run_unit(i)` round robin). The sample size is set
    from the warm-up so that the timed steps together take about `args.cpu_seconds`.
    Returns (units per second, measured ms per step, units per step, timed units)."""
    i = 0
    t0 = time.perf_counter()
    for _ in range(max(1, args.warmup)):
        run_unit(i)
        i += 1
    rate = max(1, args.warmup) / (time.perf_counter() - t0)
    per_step = max(0.2, args.cpu_seconds / max(1, args.steps))
    n = max(1, int(round(rate * per_step)))
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        for _ in range(n):
            run_unit(i)
            i += 1
        times.append(time.perf_counter() - t0)
    total = sum(times)
    return n * args.steps / total, 1000.0 * total / args.steps, n, n * args.steps


def run_reference(args):
    rank, world, local = dist_env()
    if rank != 0:
        return 0
    import numpy as np

    from paper_2606_21848_gb300.workloads import WORKLOADS, bf16_bits, generate

    import oracle
    wl = workload_of(args)
    x = generate(wl)
    if wl.q_len > 0:
        return run_reference_prefill(args, wl, x)
    if wl.latent_dim > 0:
        return run_reference_latent(args, wl, x)
    q, w, v = bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"])
    bt, sl = x["block_table"].numpy(), x["seq_lens"].numpy()
    B, Hq, D = x["q"].shape
    scale = 1.0 / math.sqrt(D)
    oracle.build()

    def one_sequence(i):
        heads = np.array([(i % B, h) for h in range(Hq)], np.int32)
        if args.standard:
            oracle.standard_decode(q, v, v, bt, sl, scale=scale, heads=heads)
        else:
            oracle.decode(q, w, v, bt, sl, scale=scale, heads=heads)

    value, ms, n, total = reference_steps(one_sequence, args)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": decode_config(wl, x, args, args.gpus),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": oracle.threads(),
                         "kind": "oracle",
                         "sample": f"each step: {n} whole sequences (all {Hq} heads, decode "
                                   f"only, fp64) of {wl.name}, round robin; {total} timed"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def workload_of(args):
    """The selected workload with the command line's overrides."""
    from paper_2606_21848_gb300.workloads import WORKLOADS
    wl = WORKLOADS[args.workload]
    if args.wr_per_query_head:
        wl = wl.with_(wr_per_query_head=True)
    if args.num_seqs > 0:
        wl = wl.with_(num_seqs=args.num_seqs)
    return wl


def decode_config(wl, x, args, world) -> dict:
    """The workload a decode line measures (the same keys and values for both arms)."""
    B, Hq, D = x["q"].shape
    Hkv, P = x["v_cache"].shape[1], x["v_cache"].shape[2]
    return {"workload": wl.name, "num_seqs": B, "q_heads": Hq, "kv_heads": Hkv,
            "head_dim": D, "page_size": P, "seq_len": wl.seq_len or list(wl.seq_len_range),
            "context_tokens": int(x["seq_lens"].sum()),
            "cache": "fp8 e4m3 + fp32 row scale" if args.fp8_cache else "bf16",
            "decode": "standard K+V (comparison)" if args.standard else
                      "keyless, composed query (x W^Q W^R)" if args.fused_query else "keyless",
            "w_r": "per query head" if wl.wr_per_query_head else "per value head",
            "l2": "GPU arm: flushed between timed steps (512 MiB write, then read back)",
            "parallelism": f"replicas x{world}"}


# ----------------------------------------------------------------------------- GPU arm --

def run_ours(args):
    import torch

    import paper_2606_21848_gb300 as kl
    from paper_2606_21848_gb300.workloads import WORKLOADS, generate

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("nccl", rank=rank, world_size=world)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    kl.load()

    wl = workload_of(args)
    from paper_2606_21848_gb300.multi import job_throughput, max_over_ranks, replica_seed
    x = generate(wl, seed=replica_seed(wl.seed, rank))   # replicas: each rank its own batch
    if wl.q_len > 0:
        return run_prefill(args, wl, x, dev, rank, world)
    if wl.latent_dim > 0:
        return run_latent(args, wl, x, dev, rank, world)
    B, Hq, D = x["q"].shape
    num_pages, Hkv, P, _ = x["v_cache"].shape
    max_pages = x["block_table"].shape[1]
    sh = kl.make_shape(B, Hq, Hkv, D, P, num_pages, max_pages, wl.wr_per_query_head)
    kernel = {"auto": kl.KL_KERNEL_AUTO, "tensor": kl.KL_KERNEL_TENSOR,
              "simt": kl.KL_KERNEL_SIMT}[args.kernel]
    splits_req = wl.num_splits if args.num_splits < 0 else args.num_splits
    S = kl.kl_decode_num_splits(sh, splits_req)

    g = {k: x[k].to(dev) for k in ("q", "w_r", "v_cache", "block_table", "seq_lens",
                                    "positions", "v_new")}
    k_cache = None
    if args.standard:
        # K = V (W^R)^T per value head, so the comparison computes the same attention.
        k_cache = torch.empty_like(g["v_cache"])
        for h in range(Hkv):
            w = g["w_r"][h].float()
            k_cache[:, h] = (g["v_cache"][:, h].float() @ w.t()).to(torch.bfloat16)
    out = torch.empty(B, Hq, D, dtype=torch.bfloat16, device=dev)
    part_o = torch.empty(B, Hq, S, D, dtype=torch.float32, device=dev)
    part_ml = torch.empty(B, Hq, S, 2, dtype=torch.float32, device=dev)
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, splits_req)), dtype=torch.uint8,
                     device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    flush_sink = torch.empty((), dtype=torch.float32, device=dev)

    def flush_l2():
        # Evict the cache rows from L2: write 512 MiB (4x L2), then read it back so that the
        # lines left in L2 are clean and their write-back does not land inside the next step.
        flush.zero_()
        torch.sum(flush, dim=0, out=flush_sink)

    stream = torch.cuda.current_stream(dev)
    opts_states = kl.decode_options(S, kernel, part_o, part_ml)
    opts_full = kl.decode_options(S, kernel)

    tc = kernel != kl.KL_KERNEL_SIMT and kl.kl_decode_kernel_available(sh, kl.KL_KERNEL_TENSOR,
                                                                      args.standard)
    # the tensor-core kernel merges the split states itself (ring-staged, any S up to the
    # library's limit); the CUDA-core kernel leaves them to the combine kernel
    one_kernel = S == 1 or tc or args.fp8_cache

    if args.fp8_cache:
        codes = torch.empty(g["v_cache"].shape, dtype=torch.uint8, device=dev)
        scales = torch.empty(g["v_cache"].shape[:-1], dtype=torch.float32, device=dev)
        kl.kl_quantize_cache_fp8(sh, g["v_cache"], codes, scales, stream)
        del g["v_cache"]
        torch.cuda.synchronize()

    def decode_call(opts, o, w, d=None):
        d = d or g
        if args.fp8_cache:
            kl.kl_decode_step_fp8(sh, d["q"], None if args.fused_query else g["w_r"], d["v_new"],
                                  d["positions"], codes, scales, d["block_table"], d["seq_lens"],
                                  S, o, kl.KL_BF16, w, err, stream)
        elif args.standard:
            kl.kl_standard_decode(sh, g["q"], k_cache, g["v_cache"], g["block_table"],
                                  g["seq_lens"], opts, o, kl.KL_BF16, w, err, stream)
        else:
            kl.kl_decode_step(sh, g["q"], None if args.fused_query else g["w_r"], g["v_new"],
                              g["positions"], g["v_cache"], g["block_table"], g["seq_lens"], opts,
                              o, kl.KL_BF16, w, err, stream)

    def step_timed(ev):
        # [append +] decode kernel | combine, bracketed by events on the launching stream; the
        # kernels are the ones kl_decode_step launches (the K+V comparison appends nothing)
        ev[0].record(stream)
        if one_kernel:
            # no middle event: two back-to-back event records alone read about 2 us apart
            decode_call(opts_full, out, ws)
        else:
            decode_call(opts_states, None, None)
            ev[1].record(stream)
            kl.kl_combine(sh, part_o, part_ml, S, out, kl.KL_BF16, stream)
        ev[2].record(stream)

    launches_per_step = (1 + (S > 1)) if args.fp8_cache else 1 if one_kernel else 2
    E = lambda: torch.cuda.Event(enable_timing=True)
    for _ in range(args.warmup):
        flush_l2()
        step_timed([E() for _ in range(3)])
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error flags {int(err.item())}"

    evs = [[E() for _ in range(3)] for _ in range(args.steps)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        for i in range(args.steps):
            flush_l2()
            step_timed(evs[i])
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    step_ms = [e[0].elapsed_time(e[2]) for e in evs]
    dec_ms = [e[0].elapsed_time(e[2] if one_kernel else e[1]) for e in evs]
    comb_ms = [0.0 if one_kernel else e[1].elapsed_time(e[2]) for e in evs]
    mean_step = statistics.mean(step_ms)
    mean_dec = statistics.mean(dec_ms)
    mean_step, mean_dec = max_over_ranks([mean_step, mean_dec], device=dev)
    assert int(err.item()) == 0, f"device error flags {int(err.item())}"

    ab = algorithmic_bytes(x, args.standard, with_wr=not args.fused_query, fp8=args.fp8_cache)
    value = job_throughput(B, world, mean_step / 1e3)
    peak, peak_kind = measured_peaks()
    dec_gbs = ab["total"] / (mean_dec / 1e3) / 1e9
    step_gbs = ab["total"] / (mean_step / 1e3) / 1e9

    # ---- end to end through the public API with host buffers ----
    e2e = None
    if not args.no_e2e:
        # the step's inputs in one pinned buffer, one host-to-device copy per step
        h_stage, d_stage, d_in = stage_inputs(
            x, ("q", "v_new", "positions", "seq_lens", "block_table"), dev)
        h_out = torch.empty(B, Hq, D, dtype=torch.bfloat16).pin_memory()
        h2d = h_stage.numel()
        d2h = h_out.numel() * h_out.element_size()

        def e2e_step():
            d_stage.copy_(h_stage, non_blocking=True)
            if args.fp8_cache:
                decode_call(opts_full, out, ws, d_in)
            elif args.standard:
                kl.kl_standard_decode(sh, d_in["q"], k_cache, g["v_cache"], d_in["block_table"],
                                      d_in["seq_lens"], opts_full, out, kl.KL_BF16, ws, err,
                                      stream)
            else:
                kl.kl_decode_step(sh, d_in["q"], None if args.fused_query else g["w_r"],
                                  d_in["v_new"], d_in["positions"],
                                  g["v_cache"], d_in["block_table"], d_in["seq_lens"], opts_full,
                                  out, kl.KL_BF16, ws, err, stream)
            h_out.copy_(out, non_blocking=True)

        for _ in range(args.warmup):
            flush_l2()
            e2e_step()
        torch.cuda.synchronize()
        ts = []
        for _ in range(args.steps):
            flush_l2()
            a, b = E(), E()
            a.record(stream)
            e2e_step()
            b.record(stream)
            ts.append((a, b))
        torch.cuda.synchronize()
        e2e_ms = statistics.mean(a.elapsed_time(b) for a, b in ts)
        e2e_ms, = max_over_ranks([e2e_ms], device=dev)
        e2e = {"value": B * world / (e2e_ms / 1e3), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms}

    sweep = None
    if (world == 1 and not args.no_sweep and args.workload == DEFAULT_WORKLOAD and
            not (args.standard or args.fp8_cache or args.fused_query or args.wr_per_query_head
                 or args.num_seqs or args.num_splits >= 0 or args.kernel != "auto")):
        sweep = sweep_workloads(args, dev, stream, flush_l2, x, g, sh, mean_dec)

    if rank != 0:
        return 0

    cpu = None
    if world == 1:
        rate, n, el = cpu_oracle_rate(x, args.cpu_seconds, args.standard)
        import oracle
        cpu = {"value": rate, "unit": "tokens/s", "cores": oracle.threads(), "kind": "oracle",
               "sample": f"{n} whole sequences of {wl.name} (all {Hq} heads, decode only, "
                         f"fp64) in {el:.1f}s"}
        r1, n1, el1, c1 = cpu_oracle_one_core(x, min(args.cpu_seconds, 5.0), args.standard)
        cpu["one_core"] = {"value": r1, "unit": "tokens/s", "cores": c1,
                           "sample": f"{n1} whole sequences (the first 4 of the batch, round "
                                     f"robin) in {el1:.1f}s"}

    kname = "tensor-fp8" if args.fp8_cache else "tensor" if tc else "simt"
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": mean_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; inputs resident in HBM)",
        "config": decode_config(wl, x, args, world),
        "launch": {"num_splits": S, "kernel": kname},
        "hbm_gbs_step": step_gbs,
        "pct_of_8tbs_step": 100.0 * step_gbs / NOMINAL_HBM_GBS,
        "ms_breakdown": {"decode": mean_dec, "combine": statistics.mean(comb_ms)},
        "kernels_per_step": launches_per_step,
        "roofline": {"bound": "hbm", "achieved": dec_gbs, "peak": peak, "unit": "GB/s",
                     "frac": dec_gbs / peak, "peak_kind": peak_kind,
                     "pct_of_8tbs": 100.0 * dec_gbs / NOMINAL_HBM_GBS,
                     "algorithmic_bytes": ab["total"],
                     "traffic": recorded_traffic(wl.name, kname)},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk.summary(),
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    if sweep is not None:
        line.update(sweep)
    print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def time_device(step, args, stream, flush_l2):
    """Mean CUDA-event time (ms) of `step()` on `stream` over args.steps timed steps after
    args.warmup untimed ones, L2 flushed before every step."""
    import torch
    E = lambda: torch.cuda.Event(enable_timing=True)
    for _ in range(args.warmup):
        flush_l2()
        step()
    torch.cuda.synchronize()
    evs = [(E(), E()) for _ in range(args.steps)]
    for a, b in evs:
        flush_l2()
        a.record(stream)
        step()
        b.record(stream)
    torch.cuda.synchronize()
    return statistics.mean(a.elapsed_time(b) for a, b in evs)


def sweep_workloads(args, dev, stream, flush_l2, x70, g70, sh70, keyless_ms):
    """The other workloads, measured in the same process with the same timing (L2 flushed
    before every step, CUDA events on the launching stream): the four other decode workloads
    (one step = kl_decode_step), the same-design K+V decode on the default batch against the
    keyless decode of the same batch, the FP8 value cache on the default batch, the latent
    value-only cache and the chunked prefill."""
    import torch

    import paper_2606_21848_gb300 as kl
    from paper_2606_21848_gb300.workloads import EXTRA, ORDER, WORKLOADS, generate

    peak, peak_kind = measured_peaks()
    launches = 0
    err = torch.zeros(1, dtype=torch.int32, device=dev)

    def gbs_entry(ms, nbytes, B, extra):
        gbs = nbytes / (ms / 1e3) / 1e9
        e = {"ms": ms, "tokens_per_s": B / (ms / 1e3), "gb_s": gbs, "frac": gbs / peak,
             "pct_of_8tbs": 100.0 * gbs / NOMINAL_HBM_GBS, "algorithmic_bytes": nbytes}
        e.update(extra)
        return e

    workloads = {}
    for name in ORDER + EXTRA:
        if name == DEFAULT_WORKLOAD:
            continue
        wl = WORKLOADS[name]
        x = generate(wl)
        B, Hq, D = x["q"].shape
        num_pages, Hkv, P, _ = x["v_cache"].shape
        sh = kl.make_shape(B, Hq, Hkv, D, P, num_pages, x["block_table"].shape[1])
        g = {k: x[k].to(dev) for k in ("q", "w_r", "v_cache", "block_table", "seq_lens",
                                        "positions", "v_new")}
        out = torch.empty(B, Hq, D, dtype=torch.bfloat16, device=dev)
        plans = [("", wl.num_splits)] + ([("auto_plan", 0)] if wl.num_splits else [])
        for suffix, req in plans:
            S = kl.kl_decode_num_splits(sh, req)
            ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, req)), dtype=torch.uint8,
                             device=dev)
            opts = kl.decode_options(req)
            tc = bool(kl.kl_decode_kernel_available(sh, kl.KL_KERNEL_TENSOR, False))

            def step():
                kl.kl_decode_step(sh, g["q"], g["w_r"], g["v_new"], g["positions"], g["v_cache"],
                                  g["block_table"], g["seq_lens"], opts, out, kl.KL_BF16, ws, err,
                                  stream)

            ms = time_device(step, args, stream, flush_l2)
            n_launch = 1 if (tc or S == 1) else 2
            launches += n_launch * args.steps
            ab = algorithmic_bytes(x, False)
            workloads[name + ("_" + suffix if suffix else "")] = gbs_entry(
                ms, ab["total"], B, {"num_splits": S, "kernel": "tensor" if tc else "simt",
                                     "kernels_per_step": n_launch,
                                     "context_tokens": ab["tokens"],
                                     "traffic": None if suffix else
                                     recorded_traffic(name, "tensor" if tc else "simt")})
        del g, out, ws, x
        torch.cuda.empty_cache()

    # The K+V comparison: the same kernel reading a K tile and a V tile per 128 tokens, with
    # K = V (W^R)^T so that it computes the same attention, against the keyless decode (without
    # the append) of the same batch.
    B, Hq, D = x70["q"].shape
    Hkv = x70["v_cache"].shape[1]
    out = torch.empty(B, Hq, D, dtype=torch.bfloat16, device=dev)
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh70, 0)), dtype=torch.uint8, device=dev)
    opts = kl.decode_options(0)
    keyless_no_append = time_device(
        lambda: kl.kl_decode_attention_ex(sh70, g70["q"], g70["w_r"], g70["v_cache"],
                                          g70["block_table"], g70["seq_lens"], opts, out,
                                          kl.KL_BF16, ws, err, stream), args, stream, flush_l2)
    k_cache = torch.empty_like(g70["v_cache"])
    for h in range(Hkv):
        k_cache[:, h] = (g70["v_cache"][:, h].float() @ g70["w_r"][h].float().t()).to(torch.bfloat16)
    standard = time_device(
        lambda: kl.kl_standard_decode(sh70, g70["q"], k_cache, g70["v_cache"], g70["block_table"],
                                      g70["seq_lens"], opts, out, kl.KL_BF16, ws, err, stream),
        args, stream, flush_l2)
    launches += 2 * args.steps
    del k_cache
    torch.cuda.empty_cache()
    ab_k = algorithmic_bytes(x70, False)
    ab_s = algorithmic_bytes(x70, True)
    kv = {"workload": DEFAULT_WORKLOAD,
          "keyless_decode": gbs_entry(keyless_no_append, ab_k["total"] - B * Hkv * D * 4, B, {"what": "kl_decode_attention (no append)"}),
          "standard_kv_decode": gbs_entry(standard, ab_s["total"], B,
                                          {"what": "kl_standard_decode, K = V (W^R)^T"}),
          "time_ratio_standard_over_keyless": standard / keyless_no_append,
          "cache_bytes_ratio": ab_s["cache"] / ab_k["cache"]}

    # The FP8 value cache of the default batch (codes + one fp32 scale per row), quantized
    # once on the GPU; one step = kl_decode_step_fp8 (the quantizing append inside the decode).
    codes = torch.empty(g70["v_cache"].shape, dtype=torch.uint8, device=dev)
    scales = torch.empty(g70["v_cache"].shape[:-1], dtype=torch.float32, device=dev)
    kl.kl_quantize_cache_fp8(sh70, g70["v_cache"], codes, scales, stream)
    S8 = kl.kl_decode_num_splits(sh70, 0)
    ws8 = torch.zeros(max(256, kl.kl_decode_workspace_size(sh70, 0)), dtype=torch.uint8,
                      device=dev)
    fp8_ms = time_device(
        lambda: kl.kl_decode_step_fp8(sh70, g70["q"], g70["w_r"], g70["v_new"], g70["positions"],
                                      codes, scales, g70["block_table"], g70["seq_lens"], 0, out,
                                      kl.KL_BF16, ws8, err, stream), args, stream, flush_l2)
    launches += (1 + (S8 > 1)) * args.steps
    del codes, scales, ws8
    torch.cuda.empty_cache()
    ab8 = algorithmic_bytes(x70, False, fp8=True)
    fp8 = gbs_entry(fp8_ms, ab8["total"], B, {"workload": DEFAULT_WORKLOAD,
                                              "what": "kl_decode_step_fp8",
                                              "speedup_over_bf16_step": keyless_ms / fp8_ms,
                                              "traffic": recorded_traffic(DEFAULT_WORKLOAD,
                                                                          "tensor-fp8")})

    # Latent value-only cache: one step = kl_latent_decode_step (three kernels).
    wl = WORKLOADS["latent_serving"]
    x = generate(wl)
    B, Hq, D = x["q"].shape
    num_pages, Hl, P, r = x["v_lat"].shape
    lsh = kl.make_latent_shape(B, Hq, Hl, D, r, P, num_pages, x["block_table"].shape[1])
    g = {k: x[k].to(dev) for k in ("q", "w_r", "w_post", "v_lat", "block_table", "seq_lens",
                                    "positions", "v_new")}
    lout = torch.empty(B, Hq, D, dtype=torch.bfloat16, device=dev)
    lws = torch.zeros(kl.kl_latent_workspace_size(lsh, 0), dtype=torch.uint8, device=dev)
    lat_ms = time_device(
        lambda: kl.kl_latent_decode_step(lsh, g["q"], g["w_r"], g["w_post"], g["v_new"],
                                         g["positions"], g["v_lat"], g["block_table"],
                                         g["seq_lens"], 0, lout, kl.KL_BF16, lws, err, stream),
        args, stream, flush_l2)
    launches += 3 * args.steps
    latent = gbs_entry(lat_ms, latent_bytes(x)["total"], B,
                       {"workload": wl.name, "what": "kl_latent_decode_step"})
    del g, lout, lws, x
    torch.cuda.empty_cache()

    # Chunked prefill: one step = kl_append_v_chunk + kl_prefill_attention; useful FLOPs of the
    # prefill kernel against the measured bf16 peak.
    wl = WORKLOADS["prefill_chunked_gqa"]
    x = generate(wl)
    T, Hq, D = x["q_chunk"].shape
    B = x["seq_lens"].shape[0]
    num_pages, Hkv, P, _ = x["v_cache"].shape
    psh = kl.make_shape(B, Hq, Hkv, D, P, num_pages, x["block_table"].shape[1])
    g = {k: x[k].to(dev) for k in ("q_chunk", "v_chunk", "w_r", "v_cache", "block_table",
                                    "seq_lens", "cu_q")}
    pout = torch.empty(T, Hq, D, dtype=torch.bfloat16, device=dev)
    max_q = int(x["q_lens"].max())
    pre_ms = time_device(
        lambda: kl.kl_prefill_attention(psh, g["q_chunk"], g["w_r"], g["v_cache"],
                                        g["block_table"], g["seq_lens"], g["cu_q"], T, max_q,
                                        pout, kl.KL_BF16, err, stream), args, stream, flush_l2)
    launches += args.steps
    fl = prefill_flops(x)
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            tpeak = float(json.load(f)["bf16_tflops"])
    except Exception:
        tpeak = 1900.0
    tfl = fl["total"] / (pre_ms / 1e3) / 1e12
    prefill = {"workload": wl.name, "what": "kl_prefill_attention", "ms": pre_ms,
               "query_tokens_per_s": T / (pre_ms / 1e3), "useful_tflops": tfl,
               "frac_of_bf16_peak": tfl / tpeak, "bf16_peak_tflops": tpeak,
               "note": "scores from hi + lo bf16 query operands, output from fp16 weights and "
                       "values: 1.5x the useful MMA work issued"}
    del g, pout, x
    torch.cuda.empty_cache()

    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error flags {int(err.item())} in the sweep"
    return {"workloads": workloads, "kv_comparison": kv, "fp8_cache": fp8, "latent": latent,
            "prefill": prefill, "sweep_gpu_launches": launches,
            "sweep_timing": "each entry: mean of --steps CUDA-event-timed steps after --warmup, "
                            "L2 flushed before every step, in this process"}


# --------------------------------------------------------------------------- prefill ----

PREFILL_METRIC = "prefill attention query tokens/s and TFLOP/s on 1 GB300"


def prefill_flops(x) -> dict:
    """Useful FLOPs of a chunked prefill: 4 D per (query row, head, visible token) -- the score
    and the output accumulation, 2 FLOPs each per dimension -- plus the routing projection,
    2 D^2 per (query row, head). The kernel issues twice the attention MMA work (hi/lo pairs)."""
    D = x["q_chunk"].shape[2]
    Hq = x["q_chunk"].shape[1]
    pairs = 0
    for L, n in zip(x["seq_lens"].tolist(), x["q_lens"].tolist()):
        # row i at position L - n + i sees L - n + i + 1 tokens
        pairs += n * (L - n) + n * (n + 1) // 2
    T = int(x["cu_q"][-1])
    attn = 4.0 * D * Hq * pairs
    route = 2.0 * T * Hq * D * D
    return {"attention": attn, "routing": route, "total": attn + route, "pairs": pairs, "rows": T}


def cpu_oracle_prefill_rate(x, seconds: float):
    """Time the fp64 oracle (as it stands) on query rows (all heads) spread over the chunk."""
    import numpy as np

    import oracle
    from paper_2606_21848_gb300.workloads import bf16_bits

    q, w, v = bf16_bits(x["q_chunk"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"])
    bt, sl, cu = x["block_table"].numpy(), x["seq_lens"].numpy(), x["cu_q"].numpy()
    T, Hq, D = x["q_chunk"].shape
    wr_pq = bool(x["workload"].wr_per_query_head)
    oracle.build()
    stride = 7919                       # a fixed walk over the rows, early and late positions
    rows, r = 0, 0
    t0 = time.perf_counter()
    while True:
        sel = np.array([(r, h) for h in range(Hq)], np.int32)
        oracle.prefill(q, w, v, bt, sl, cu, scale=1.0 / math.sqrt(D), wr_per_query_head=wr_pq,
                       rows=sel)
        rows += 1
        r = (r + stride) % T
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    return rows / el, rows, el


def run_reference_prefill(args, wl, x):
    import numpy as np

    import oracle
    from paper_2606_21848_gb300.workloads import bf16_bits

    q, w, v = bf16_bits(x["q_chunk"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"])
    bt, sl, cu = x["block_table"].numpy(), x["seq_lens"].numpy(), x["cu_q"].numpy()
    T, Hq, D = x["q_chunk"].shape
    wr_pq = bool(wl.wr_per_query_head)
    oracle.build()
    stride = 7919                       # a fixed walk over the rows, early and late positions

    def one_row(i):
        sel = np.array([((i * stride) % T, h) for h in range(Hq)], np.int32)
        oracle.prefill(q, w, v, bt, sl, cu, scale=1.0 / math.sqrt(D), wr_per_query_head=wr_pq,
                       rows=sel)

    value, ms, n, total = reference_steps(one_row, args)
    B = x["seq_lens"].shape[0]
    num_pages, Hkv, P, _ = x["v_cache"].shape
    line = {
        "impl": "reference", "metric": PREFILL_METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": prefill_config(wl, x, args.gpus),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": oracle.threads(),
                         "kind": "oracle",
                         "sample": f"each step: {n} query rows (all {Hq} heads, fp64) of "
                                   f"{wl.name} on a fixed stride over the chunk; {total} timed"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def prefill_config(wl, x, world) -> dict:
    T, Hq, D = x["q_chunk"].shape
    B = x["seq_lens"].shape[0]
    Hkv, P = x["v_cache"].shape[1], x["v_cache"].shape[2]
    return {"workload": wl.name, "num_seqs": B, "q_heads": Hq, "kv_heads": Hkv,
            "head_dim": D, "page_size": P, "seq_len": wl.seq_len, "chunk": wl.q_len,
            "query_rows": T, "visible_pairs": prefill_flops(x)["pairs"],
            "w_r": "per query head" if wl.wr_per_query_head else "per value head",
            "l2": "GPU arm: flushed between timed steps (512 MiB write, then read back)",
            "parallelism": f"replicas x{world}"}


def run_prefill(args, wl, x, dev, rank, world):
    """One prefill step = the chunk append (kl_append_v_chunk) + the chunked prefill
    (kl_prefill_attention), inputs resident in HBM, L2 flushed between steps."""
    import torch

    import paper_2606_21848_gb300 as kl
    from paper_2606_21848_gb300.multi import job_throughput, max_over_ranks

    T, Hq, D = x["q_chunk"].shape
    B = x["seq_lens"].shape[0]
    num_pages, Hkv, P, _ = x["v_cache"].shape
    sh = kl.make_shape(B, Hq, Hkv, D, P, num_pages, x["block_table"].shape[1],
                       wl.wr_per_query_head)
    max_q = int(x["q_lens"].max())
    g = {k: x[k].to(dev) for k in ("q_chunk", "v_chunk", "w_r", "v_cache", "block_table",
                                    "seq_lens", "cu_q")}
    out = torch.empty(T, Hq, D, dtype=torch.bfloat16, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    flush_sink = torch.empty((), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def flush_l2():
        flush.zero_()
        torch.sum(flush, dim=0, out=flush_sink)

    def step(d, ev=None):
        if ev: ev[0].record(stream)
        kl.kl_append_v_chunk(sh, d["v_chunk"], d["block_table"], d["seq_lens"], d["cu_q"], T,
                             max_q, g["v_cache"], err, stream)
        if ev: ev[1].record(stream)
        kl.kl_prefill_attention(sh, d["q_chunk"], g["w_r"], g["v_cache"], d["block_table"],
                                d["seq_lens"], d["cu_q"], T, max_q, out, kl.KL_BF16, err, stream)
        if ev: ev[2].record(stream)

    E = lambda: torch.cuda.Event(enable_timing=True)
    for _ in range(args.warmup):
        flush_l2()
        step(g, [E(), E(), E()])
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error flags {int(err.item())}"
    evs = [[E(), E(), E()] for _ in range(args.steps)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(dev.index) as clk:
        for i in range(args.steps):
            flush_l2()
            step(g, evs[i])
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    step_ms = statistics.mean(e[0].elapsed_time(e[2]) for e in evs)
    app_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    pre_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
    step_ms, app_ms, pre_ms = max_over_ranks([step_ms, app_ms, pre_ms], device=dev)
    assert int(err.item()) == 0, f"device error flags {int(err.item())}"

    fl = prefill_flops(x)
    tflops = fl["total"] / (pre_ms / 1e3) / 1e12
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peak, peak_kind = float(json.load(f)["bf16_tflops"]), "measured (cuBLAS bf16 burst)"
    except Exception:
        peak, peak_kind = 1900.0, "fallback"

    e2e = None
    if not args.no_e2e:
        # the step's inputs in one pinned buffer, one host-to-device copy per step
        h_stage, d_stage, d_in = stage_inputs(
            x, ("q_chunk", "v_chunk", "block_table", "seq_lens", "cu_q"), dev)
        h_out = torch.empty(T, Hq, D, dtype=torch.bfloat16).pin_memory()
        h2d = h_stage.numel()
        d2h = h_out.numel() * h_out.element_size()

        def e2e_step():
            d_stage.copy_(h_stage, non_blocking=True)
            step(d_in)
            h_out.copy_(out, non_blocking=True)

        for _ in range(args.warmup):
            flush_l2()
            e2e_step()
        torch.cuda.synchronize()
        ts = []
        for _ in range(args.steps):
            flush_l2()
            a, b = E(), E()
            a.record(stream)
            e2e_step()
            b.record(stream)
            ts.append((a, b))
        torch.cuda.synchronize()
        e2e_ms = statistics.mean(a.elapsed_time(b) for a, b in ts)
        e2e_ms, = max_over_ranks([e2e_ms], device=dev)
        e2e = {"value": T * world / (e2e_ms / 1e3), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms}

    if rank != 0:
        return 0
    cpu = None
    if world == 1:
        import oracle
        rate, n, el = cpu_oracle_prefill_rate(x, args.cpu_seconds)
        cpu = {"value": rate, "unit": "tokens/s", "cores": oracle.threads(), "kind": "oracle",
               "sample": f"{n} query rows (all {Hq} heads) of {wl.name} on a fixed stride over "
                         f"the chunk, fp64, in {el:.1f}s"}
    line = {
        "metric": PREFILL_METRIC, "value": job_throughput(T, world, step_ms / 1e3), "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; inputs resident in HBM)",
        "config": prefill_config(wl, x, world),
        "operands": "scores: hi + lo bf16 query against the bf16 tile; output: fp16 weights "
                    "against the tile converted to fp16 (1.5x the attention MMA work)",
        "ms_breakdown": {"append": app_ms, "prefill": pre_ms},
        "tflops": tflops,
        "kernels_per_step": 2,
        "roofline": {"bound": "tensor", "achieved": tflops, "peak": peak, "unit": "TFLOP/s",
                     "frac": tflops / peak, "peak_kind": peak_kind,
                     "algorithmic_flops": fl["total"], "traffic": None},
        "gpu_launches": 2 * args.steps,
        "clocks": clk.summary(),
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


# ---------------------------------------------------------------------------- latent ----

LATENT_METRIC = ("latent value-only cache decode tokens/s and achieved HBM GB/s "
                 "(% of 8 TB/s) on 1 GB300")


def latent_bytes(x) -> dict:
    """Bytes a latent decode step must move once: the latent rows, W^R, W_post, q, out, the
    block table, and the appended latent row (read and written)."""
    B, Hq, D = x["q"].shape
    num_pages, Hl, P, r = x["v_lat"].shape
    tokens = int(x["seq_lens"].sum())
    lat = tokens * Hl * r * 2
    w = x["w_r"].numel() * 2 + x["w_post"].numel() * 2
    io = 2 * B * Hq * D * 2
    bt = sum(math.ceil(int(L) / P) for L in x["seq_lens"].tolist()) * 4 + B * 4
    append = 2 * B * Hl * r * 2
    return {"latent": lat, "total": lat + w + io + bt + append, "tokens": tokens}


def cpu_oracle_latent_rate(x, seconds: float):
    import numpy as np

    import oracle
    from paper_2606_21848_gb300.workloads import bf16_bits
    q, w, wp, v = (bf16_bits(x[k]) for k in ("q", "w_r", "w_post", "v_lat"))
    bt, sl = x["block_table"].numpy(), x["seq_lens"].numpy()
    B, Hq, D = x["q"].shape
    r = x["v_lat"].shape[3]
    oracle.build()
    seqs, b = 0, 0
    t0 = time.perf_counter()
    while True:
        heads = np.array([(b, h) for h in range(Hq)], np.int32)
        oracle.latent_decode(q, w, wp, v, bt, sl, scale=1.0 / math.sqrt(r), heads=heads)
        seqs += 1
        b = (b + 1) % B
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    return seqs / el, seqs, el


def run_reference_latent(args, wl, x):
    import numpy as np

    import oracle
    from paper_2606_21848_gb300.workloads import bf16_bits
    q, w, wp, v = (bf16_bits(x[k]) for k in ("q", "w_r", "w_post", "v_lat"))
    bt, sl = x["block_table"].numpy(), x["seq_lens"].numpy()
    B, Hq, D = x["q"].shape
    r = x["v_lat"].shape[3]
    oracle.build()

    def one_sequence(i):
        heads = np.array([(i % B, h) for h in range(Hq)], np.int32)
        oracle.latent_decode(q, w, wp, v, bt, sl, scale=1.0 / math.sqrt(r), heads=heads)

    value, ms, n, total = reference_steps(one_sequence, args)
    line = {
        "impl": "reference", "metric": LATENT_METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": latent_config(wl, x, args.gpus),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": oracle.threads(),
                         "kind": "oracle",
                         "sample": f"each step: {n} whole sequences (all {Hq} heads, fp64) of "
                                   f"{wl.name}, round robin; {total} timed"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def latent_config(wl, x, world) -> dict:
    B, Hq, D = x["q"].shape
    num_pages, Hl, P, r = x["v_lat"].shape
    return {"workload": wl.name, "num_seqs": B, "q_heads": Hq, "latent_heads": Hl,
            "head_dim": D, "latent_dim": r, "page_size": P, "seq_len": wl.seq_len,
            "context_tokens": int(x["seq_lens"].sum()),
            "w_r": "per query head" if wl.wr_per_query_head else "per latent group",
            "w_post": "per query head",
            "l2": "GPU arm: flushed between timed steps (512 MiB write, then read back)",
            "parallelism": f"replicas x{world}"}


def run_latent(args, wl, x, dev, rank, world):
    """One latent decode step = kl_latent_decode_step: the current token's latent rows appended
    inside the tensor-core decode over the latent rows, between the absorbed-query and the
    expansion kernels (three launches)."""
    import torch

    import paper_2606_21848_gb300 as kl
    from paper_2606_21848_gb300.multi import job_throughput, max_over_ranks

    B, Hq, D = x["q"].shape
    num_pages, Hl, P, r = x["v_lat"].shape
    max_pages = x["block_table"].shape[1]
    lsh = kl.make_latent_shape(B, Hq, Hl, D, r, P, num_pages, max_pages, wl.wr_per_query_head)
    ash = kl.make_shape(B, Hq, Hl, r, P, num_pages, max_pages)      # the decode over latent rows
    splits_req = wl.num_splits if args.num_splits < 0 else args.num_splits
    S = kl.kl_decode_num_splits(ash, splits_req)
    g = {k: x[k].to(dev) for k in ("q", "w_r", "w_post", "v_lat", "block_table", "seq_lens",
                                    "positions", "v_new")}
    out = torch.empty(B, Hq, D, dtype=torch.bfloat16, device=dev)
    ws = torch.zeros(kl.kl_latent_workspace_size(lsh, splits_req), dtype=torch.uint8, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    flush_sink = torch.empty((), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def flush_l2():
        flush.zero_()
        torch.sum(flush, dim=0, out=flush_sink)

    def step(d, ev=None):
        if ev: ev[0].record(stream)
        kl.kl_latent_decode_step(lsh, d["q"], g["w_r"], g["w_post"], d["v_new"], d["positions"],
                                 g["v_lat"], d["block_table"], d["seq_lens"], splits_req, out,
                                 kl.KL_BF16, ws, err, stream)
        if ev: ev[1].record(stream)

    E = lambda: torch.cuda.Event(enable_timing=True)
    for _ in range(args.warmup):
        flush_l2()
        step(g, [E(), E()])
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error flags {int(err.item())}"
    evs = [[E(), E()] for _ in range(args.steps)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(dev.index) as clk:
        for i in range(args.steps):
            flush_l2()
            step(g, evs[i])
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    step_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    step_ms, = max_over_ranks([step_ms], device=dev)
    dec_ms = step_ms
    assert int(err.item()) == 0, f"device error flags {int(err.item())}"
    ab = latent_bytes(x)
    peak, peak_kind = measured_peaks()
    dec_gbs = ab["total"] / (dec_ms / 1e3) / 1e9

    e2e = None
    if not args.no_e2e:
        # the step's inputs in one pinned buffer, one host-to-device copy per step
        h_stage, d_stage, d_in = stage_inputs(
            x, ("q", "v_new", "positions", "seq_lens", "block_table"), dev)
        h_out = torch.empty(B, Hq, D, dtype=torch.bfloat16).pin_memory()
        h2d = h_stage.numel()
        d2h = h_out.numel() * h_out.element_size()

        def e2e_step():
            d_stage.copy_(h_stage, non_blocking=True)
            step(d_in)
            h_out.copy_(out, non_blocking=True)

        for _ in range(args.warmup):
            flush_l2()
            e2e_step()
        torch.cuda.synchronize()
        ts = []
        for _ in range(args.steps):
            flush_l2()
            a, b = E(), E()
            a.record(stream)
            e2e_step()
            b.record(stream)
            ts.append((a, b))
        torch.cuda.synchronize()
        e2e_ms = statistics.mean(a.elapsed_time(b) for a, b in ts)
        e2e_ms, = max_over_ranks([e2e_ms], device=dev)
        e2e = {"value": B * world / (e2e_ms / 1e3), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms}

    if rank != 0:
        return 0
    cpu = None
    if world == 1:
        import oracle
        rate, n, el = cpu_oracle_latent_rate(x, args.cpu_seconds)
        cpu = {"value": rate, "unit": "tokens/s", "cores": oracle.threads(), "kind": "oracle",
               "sample": f"{n} whole sequences of {wl.name} (all {Hq} heads, fp64) in {el:.1f}s"}
    line = {
        "metric": LATENT_METRIC, "value": job_throughput(B, world, step_ms / 1e3), "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; inputs resident in HBM)",
        "config": latent_config(wl, x, world),
        "launch": {"num_splits": S},
        "ms_breakdown": {"latent_decode_step": step_ms},
        "kernels_per_step": 3,
        "roofline": {"bound": "hbm", "achieved": dec_gbs, "peak": peak, "unit": "GB/s",
                     "frac": dec_gbs / peak, "peak_kind": peak_kind,
                     "pct_of_8tbs": 100.0 * dec_gbs / NOMINAL_HBM_GBS,
                     "algorithmic_bytes": ab["total"],
                     "timed": "the kl_latent_decode_step call (absorbed query, decode with the "
                              "fused append, expansion)",
                     "traffic": recorded_traffic(wl.name, "tensor"),
                     "traffic_of": "the decode kernel over the latent rows (ncu)"},
        "gpu_launches": 3 * args.steps,
        "clocks": clk.summary(),
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
