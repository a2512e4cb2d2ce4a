"""GPU parity: the CUDA path through the C ABI against the fp64 oracle on seeded inputs.

Bar: bit-exact for the append (page/row indexing) and for block-table permutations at a fixed
split plan; |gpu - oracle| <= 2e-3 + 1e-2 |oracle| elementwise for every floating-point output.
"""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300.workloads import WORKLOADS, Workload, bf16_bits, generate
from tests import _gpu
from tests._gpu import KERNELS, assert_parity, decode, oracle_decode, shape_of, to_dev
from tests._inputs import tiny

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    kl.build()
    kl.load()


def _tc_available(x, standard=False) -> bool:
    """Whether the tensor-core kernel accepts this geometry (asks the library)."""
    return kl.kl_decode_kernel_available(shape_of(x), kl.KL_KERNEL_TENSOR, standard)


def _kernel_or_skip(kname, x, standard=False):
    if kname == "tensor" and not _tc_available(x, standard):
        pytest.skip("tensor-core kernel does not support this geometry")
    return KERNELS[kname]


# ---------------------------------------------------------------- append (bit-exact) -----

@pytest.mark.parametrize("D,P,Hkv", [(64, 16, 4), (128, 16, 8), (128, 32, 8)])
def test_append_is_bit_exact(D, P, Hkv):
    x = tiny(B=4, Hq=2 * Hkv, Hkv=Hkv, D=D, P=P, lens=(1, P, 3 * P + 5, 7 * P))
    g = to_dev(x)
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    kl.kl_append_v(shape_of(x), g["v_new"], g["block_table"], g["positions"], g["v_cache"], err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    want = oracle.append(bf16_bits(x["v_cache"]), bf16_bits(x["v_new"]), x["block_table"].numpy(),
                         x["positions"].numpy())
    np.testing.assert_array_equal(bf16_bits(g["v_cache"].cpu()), want)


def test_append_flags_bad_position_and_page_and_skips_them():
    x = tiny(B=3, lens=(20, 40, 60))
    x["positions"] = torch.tensor([-1, 10_000, 5], dtype=torch.int32)
    x["block_table"][2, 0] = x["num_pages"] + 3          # page id outside the pool
    g = to_dev(x)
    before = bf16_bits(g["v_cache"].cpu()).copy()
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    kl.kl_append_v(shape_of(x), g["v_new"], g["block_table"], g["positions"], g["v_cache"], err)
    torch.cuda.synchronize()
    assert int(err.item()) == kl.KL_FLAG_BAD_POSITION | kl.KL_FLAG_BAD_PAGE
    np.testing.assert_array_equal(bf16_bits(g["v_cache"].cpu()), before)


# ---------------------------------------------------------------------- routing ---------

@pytest.mark.parametrize("per_q", [False, True])
def test_route_query_matches_oracle(per_q):
    x = tiny(B=3, Hq=32, Hkv=8, D=128, lens=(5, 6, 7), wr_per_query_head=per_q)
    g = to_dev(x)
    q_r = torch.empty(3, 32, 128, dtype=torch.float32, device=_gpu.dev())
    kl.kl_route_query(shape_of(x), g["q"], g["w_r"], q_r)
    torch.cuda.synchronize()
    want = oracle.route(bf16_bits(x["q"]), bf16_bits(x["w_r"]), 8, per_q)
    np.testing.assert_allclose(q_r.cpu().double().numpy(), want, rtol=1e-5, atol=1e-5)


# ----------------------------------------------------------------------- decode ---------

SHAPES = [
    dict(B=1, Hq=4, Hkv=4, D=64, P=16, lens=(256,)),                     # MHA, D 64
    dict(B=3, Hq=8, Hkv=2, D=64, P=16, lens=(1, 37, 300)),               # GQA 4, ragged tail
    dict(B=4, Hq=32, Hkv=8, D=128, P=16, lens=(0, 1, 129, 1000)),        # empty / 1 / tiles+tail
    dict(B=2, Hq=64, Hkv=8, D=128, P=32, lens=(513, 2047)),              # GQA 8, P 32
    dict(B=2, Hq=8, Hkv=8, D=128, P=16, lens=(700, 64)),                 # MHA, D 128
    dict(B=2, Hq=16, Hkv=8, D=128, P=16, lens=(333, 1280)),              # GQA 2
    dict(B=2, Hq=8, Hkv=1, D=128, P=16, lens=(1500, 9)),                 # MQA, group 8
    dict(B=2, Hq=12, Hkv=2, D=128, P=16, lens=(2222, 640)),              # Qwen2-1.5B heads, group 6
    dict(B=3, Hq=24, Hkv=8, D=128, P=64, lens=(5, 300, 1025)),           # group 3, P 64
]


@pytest.mark.parametrize("kname", ["simt", "tensor"])
@pytest.mark.parametrize("si", range(len(SHAPES)))
@pytest.mark.parametrize("splits", [1, 3, 0])
def test_decode_matches_oracle(kname, si, splits):
    x = tiny(**SHAPES[si])
    k = _kernel_or_skip(kname, x)
    out, err = decode(to_dev(x), shape_of(x), kernel=k, num_splits=splits)
    assert err == 0
    want = oracle_decode(x, _gpu.default_scale(x))
    assert_parity(out.cpu().numpy(), want, f"{kname} {SHAPES[si]} S={splits}")


# Group sizes 4 and 8 take the two compute-warp layouts of the tensor-core kernel (eight warps
# of 2 heads, four warps of 8 heads).
@pytest.mark.parametrize("kname", ["simt", "tensor"])
@pytest.mark.parametrize("G", [4, 8])
def test_decode_per_query_head_routing(kname, G):
    x = tiny(B=2, Hq=8 * G, Hkv=8, D=128, P=16, lens=(260, 999), wr_per_query_head=True)
    k = _kernel_or_skip(kname, x)
    out, err = decode(to_dev(x), shape_of(x), kernel=k, num_splits=2)
    assert err == 0
    assert_parity(out.cpu().numpy(), oracle_decode(x, _gpu.default_scale(x)), kname)


@pytest.mark.parametrize("kname", ["simt", "tensor"])
def test_decode_custom_scale_and_bf16_output(kname):
    x = tiny(B=2, Hq=16, Hkv=4, D=128, P=16, lens=(77, 400))
    k = _kernel_or_skip(kname, x)
    sh = shape_of(x, scale=0.3)
    out32, _ = decode(to_dev(x), sh, kernel=k, num_splits=2)
    out16, _ = decode(to_dev(x), sh, kernel=k, num_splits=2, out_dtype=kl.KL_BF16)
    want = oracle_decode(x, 0.3)
    assert_parity(out32.cpu().numpy(), want, "fp32 out")
    # bf16 output = the fp32 result rounded once: within half a bf16 ulp of it
    np.testing.assert_allclose(out16.float().cpu().numpy(), out32.cpu().numpy(), rtol=2 ** -8,
                               atol=1e-6)


@pytest.mark.parametrize("kname", ["simt", "tensor"])
def test_block_table_permutation_is_bit_exact(kname):
    x = tiny(B=3, Hq=32, Hkv=8, D=128, P=16, lens=(100, 555, 1024))
    k = _kernel_or_skip(kname, x)
    out1, _ = decode(to_dev(x), shape_of(x), kernel=k, num_splits=3)
    perm = torch.randperm(x["num_pages"], generator=torch.Generator().manual_seed(5))
    inv = torch.argsort(perm)
    y = dict(x)
    y["v_cache"] = x["v_cache"][perm].contiguous()
    bt = x["block_table"].clone()
    m = bt >= 0
    bt[m] = inv[bt[m].long()].to(torch.int32)
    y["block_table"] = bt
    out2, _ = decode(to_dev(y), shape_of(y), kernel=k, num_splits=3)
    assert torch.equal(out1.cpu(), out2.cpu())


@pytest.mark.parametrize("kname", ["simt", "tensor"])
def test_split_counts_agree(kname):
    """S = 1 writes the output directly; larger S are merged by the last split of each
    (sequence, value head) to finish (tensor-core kernel: direct loads up to 8 splits, staged
    through the ring beyond) or by the combine kernel (CUDA-core kernel)."""
    x = tiny(B=2, Hq=32, Hkv=8, D=128, P=16, lens=(2000, 4096))
    k = _kernel_or_skip(kname, x)
    want = oracle_decode(x, _gpu.default_scale(x))
    for s in (1, 2, 5, 8, 16, 32, 64):
        out, err = decode(to_dev(x), shape_of(x), kernel=k, num_splits=s)
        assert err == 0
        assert_parity(out.cpu().numpy(), want, f"{kname} S={s}")


@pytest.mark.parametrize("splits", [9, 17, 100, 1000])
def test_many_split_states_merged_in_the_kernel(splits):
    """One long sequence over one value head, so that every split is a CTA of its own: 9, 17,
    100 and the most (157 splits of 128 tokens) states, merged by the last CTA through the ring
    in one or several rounds of bulk copies."""
    x = tiny(B=1, Hq=4, Hkv=1, D=128, P=16, lens=(20000,), seed=24)
    want = oracle_decode(x, _gpu.default_scale(x))
    for _ in range(2):              # the counters are back at zero for the second call
        out, err = decode(to_dev(x), shape_of(x), kernel=kl.KL_KERNEL_TENSOR, num_splits=splits)
        assert err == 0
        assert_parity(out.cpu().numpy(), want, f"S={splits}")


@pytest.mark.parametrize("kname", ["simt", "tensor"])
def test_workspace_reused_across_calls_and_shapes(kname):
    """One workspace, zero-filled once, serves repeated calls and different shapes -- batch
    sizes and split counts that change from call to call, as in serving (the merge counters
    keep a front region that no split state covers) -- with identical results for identical
    inputs."""
    xa = tiny(B=2, Hq=32, Hkv=8, D=128, P=16, lens=(900, 3000), seed=21)
    xb = tiny(B=3, Hq=16, Hkv=4, D=128, P=16, lens=(129, 2500, 40), seed=22)
    xc = tiny(B=6, Hq=32, Hkv=8, D=128, P=16, lens=(3000, 2900, 2800, 100, 2000, 1500), seed=23)
    k = _kernel_or_skip(kname, xa)
    ws = torch.zeros(1 << 22, dtype=torch.uint8, device=_gpu.dev())
    outs = []
    for x, splits in ((xa, 6), (xb, 11), (xa, 6), (xc, 40), (xb, 3), (xa, 6), (xc, 7), (xa, 40)):
        g = to_dev(x)
        sh = shape_of(x)
        assert kl.kl_decode_workspace_size(sh, splits) <= ws.numel()
        out = torch.full(g["q"].shape, float("nan"), dtype=torch.float32, device=_gpu.dev())
        err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
        kl.kl_decode_attention_ex(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                                  g["seq_lens"], kl.decode_options(splits, k), out, kl.KL_FP32,
                                  ws, err)
        torch.cuda.synchronize()
        assert int(err.item()) == 0
        assert_parity(out.cpu().numpy(), oracle_decode(x, _gpu.default_scale(x)), f"S={splits}")
        outs.append(out.cpu())
    assert torch.equal(outs[0], outs[2]) and torch.equal(outs[0], outs[5])


def _step(x, kernel, num_splits, out_dtype=kl.KL_FP32):
    g = to_dev(x)
    sh = shape_of(x)
    B, Hq, D = g["q"].shape
    out = torch.full((B, Hq, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, num_splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_step(sh, g["q"], g["w_r"], g["v_new"], g["positions"], g["v_cache"],
                      g["block_table"], g["seq_lens"], kl.decode_options(num_splits, kernel), out,
                      out_dtype, ws, err)
    torch.cuda.synchronize()
    return out.cpu().numpy(), bf16_bits(g["v_cache"].cpu()), int(err.item())


@pytest.mark.parametrize("kname", ["simt", "tensor"])
@pytest.mark.parametrize("splits", [1, 3, 16])
@pytest.mark.parametrize("where", ["last", "middle", "past_end"])
def test_fused_decode_step_matches_append_then_decode(kname, splits, where):
    """kl_decode_step = kl_append_v then decode: cache bit-exact, output at tolerance."""
    x = tiny(B=3, Hq=32, Hkv=8, D=128, P=16, lens=(1, 700, 2048))
    k = _kernel_or_skip(kname, x)
    L = x["seq_lens"]
    if where == "middle":
        x["positions"] = (L // 2).to(torch.int32)
    elif where == "past_end":
        # past the sequence's end but inside its last allocated page
        x["positions"] = torch.minimum(L + 5, (L + 15) // 16 * 16 - 1).to(torch.int32)
    out, cache, err = _step(x, k, splits)
    assert err == 0
    want_cache = oracle.append(bf16_bits(x["v_cache"]), bf16_bits(x["v_new"]),
                               x["block_table"].numpy(), x["positions"].numpy())
    np.testing.assert_array_equal(cache, want_cache)
    y = dict(x)
    y["v_cache"] = torch.from_numpy(want_cache.view(np.int16)).view(torch.bfloat16)
    assert_parity(out, oracle_decode(y, _gpu.default_scale(x)), f"{kname} {where} S={splits}")


@pytest.mark.parametrize("kname", ["simt", "tensor"])
def test_fused_decode_step_flags_bad_position_and_page(kname):
    x = tiny(B=3, Hq=16, Hkv=4, D=128, P=16, lens=(40, 90, 130))
    k = _kernel_or_skip(kname, x)
    x["positions"] = torch.tensor([39, -3, 129], dtype=torch.int32)
    x["block_table"][2, 129 // 16] = -1                     # page of sequence 2's new row
    y = dict(x)
    y["block_table"] = x["block_table"].clone()
    before = bf16_bits(x["v_cache"]).copy()
    _, cache, err = _step(x, k, 1)
    assert err & kl.KL_FLAG_BAD_POSITION and err & kl.KL_FLAG_BAD_PAGE
    # only sequence 0's row changed
    want = oracle.append(before, bf16_bits(x["v_new"])[:1], x["block_table"].numpy()[:1],
                         x["positions"].numpy()[:1])
    np.testing.assert_array_equal(cache, want)


@pytest.mark.parametrize("kname", ["simt", "tensor"])
def test_bad_page_and_length_raise_flags(kname):
    x = tiny(B=2, Hq=16, Hkv=4, D=128, P=16, lens=(100, 50))
    k = _kernel_or_skip(kname, x)
    y = dict(x)
    y["block_table"] = x["block_table"].clone()
    y["block_table"][0, 2] = -7
    _, err = decode(to_dev(y), shape_of(y), kernel=k, num_splits=1)
    assert err & kl.KL_FLAG_BAD_PAGE
    z = dict(x)
    z["seq_lens"] = torch.tensor([100, 10 ** 6], dtype=torch.int32)
    out, err = decode(to_dev(z), shape_of(z), kernel=k, num_splits=1)
    assert err & kl.KL_FLAG_BAD_LENGTH
    # the valid sequence is still right
    want = oracle_decode(x, _gpu.default_scale(x))
    assert_parity(out[0].cpu().numpy(), want[0], "valid sequence next to a bad length")


# ---------------------------------------------------------------------- combine ---------

def test_combine_matches_oracle():
    rng = np.random.default_rng(7)
    B, Hq, S, D = 3, 8, 6, 128
    po = rng.standard_normal((B, Hq, S, D)).astype(np.float32)
    ml = np.stack([rng.normal(0, 3, (B, Hq, S)), rng.uniform(0.5, 50, (B, Hq, S))], -1)
    ml = ml.astype(np.float32)
    ml[0, 0, 2:, 1] = 0.0                      # empty splits
    ml[0, 0, 2:, 0] = -np.inf
    ml[1, 3, :, 1] = 0.0                       # all empty -> zeros
    ml[1, 3, :, 0] = -np.inf
    sh = kl.make_shape(B, Hq, 2, D, 16, 1, 1)
    out = torch.empty(B, Hq, D, dtype=torch.float32, device=_gpu.dev())
    kl.kl_combine(sh, torch.from_numpy(po).cuda(), torch.from_numpy(ml).cuda(), S, out, kl.KL_FP32)
    torch.cuda.synchronize()
    want = oracle.combine(po.astype(np.float64), ml.astype(np.float64))
    np.testing.assert_allclose(out.cpu().numpy(), want, rtol=1e-5, atol=1e-6)
    assert np.all(out.cpu().numpy()[1, 3] == 0)


# ------------------------------------------------------------- standard K + V -----------

@pytest.mark.parametrize("kname", ["simt", "tensor"])
@pytest.mark.parametrize("G", [4, 8])
def test_standard_kv_decode_matches_oracle(kname, G):
    x = tiny(B=3, Hq=8 * G, Hkv=8, D=128, P=16, lens=(1, 300, 1111))
    k = _kernel_or_skip(kname, x, standard=True)
    kc = torch.randn(x["v_cache"].shape, generator=torch.Generator().manual_seed(3)).to(torch.bfloat16)
    g = to_dev(x)
    out, err = decode(g, shape_of(x), kernel=k, num_splits=2, k_cache=kc.to(_gpu.dev()))
    assert err == 0
    want = oracle.standard_decode(bf16_bits(x["q"]), bf16_bits(kc), bf16_bits(x["v_cache"]),
                                  x["block_table"].numpy(), x["seq_lens"].numpy(),
                                  scale=_gpu.default_scale(x))
    assert_parity(out.cpu().numpy(), want, "standard K+V")


# ------------------------------------------------------- the five decode workloads ------

def _append_then_decode(x, kernel, num_splits):
    g = to_dev(x)
    sh = shape_of(x)
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    kl.kl_append_v(sh, g["v_new"], g["block_table"], g["positions"], g["v_cache"], err)
    out, err2 = decode(g, sh, kernel=kernel, num_splits=num_splits)
    return out, int(err.item()) | err2


def _with_appended(x):
    y = dict(x)
    y["v_cache"] = torch.from_numpy(
        oracle.append(bf16_bits(x["v_cache"]), bf16_bits(x["v_new"]), x["block_table"].numpy(),
                      x["positions"].numpy()).view(np.int16)).view(torch.bfloat16)
    return y


@pytest.mark.parametrize("kname", ["simt", "tensor"])
@pytest.mark.parametrize("name", ["tiny_mha", "small_gqa"])
def test_workload_full_parity(name, kname):
    wl = WORKLOADS[name]
    x = generate(wl)
    k = _kernel_or_skip(kname, x)
    out, err = _append_then_decode(x, k, wl.num_splits)
    assert err == 0
    want = oracle_decode(_with_appended(x), _gpu.default_scale(x))
    assert_parity(out.cpu().numpy(), want, f"{name} {kname}")


@pytest.mark.slow
@pytest.mark.parametrize("kname", ["simt", "tensor"])
@pytest.mark.parametrize("name", ["long_context", "ragged_serving", "high_concurrency_70b"])
def test_workload_sampled_parity(name, kname):
    """Full-size workloads in the bench's launch configuration; sampled heads vs the oracle."""
    wl = WORKLOADS[name]
    x = generate(wl)
    k = _kernel_or_skip(kname, x)
    out, err = _append_then_decode(x, k, wl.num_splits)
    assert err == 0
    rng = np.random.default_rng(wl.seed)
    B, Hq = wl.num_seqs, wl.num_q_heads
    heads = [(int(b), int(h)) for b, h in zip(rng.integers(0, B, 48), rng.integers(0, Hq, 48))]
    heads += [(B - 1, Hq - 1), (0, 0)]
    want = oracle_decode(_with_appended(x), _gpu.default_scale(x), heads=heads)
    got = np.stack([out[b, h].cpu().numpy() for b, h in heads])
    assert_parity(got, want, f"{name} {kname}")
    assert np.isfinite(out.cpu().numpy()).all()


# ------------------------------------------------- composed query (fused W^Q W^R) -----------

@pytest.mark.parametrize("kname", ["simt", "tensor"])
@pytest.mark.parametrize("num_splits", [1, 3, 0])
def test_composed_query_mode_matches_oracle_with_identity_routing(kname, num_splits):
    """w_r = NULL: the query already is x W^Q W^R (Section 2.1's precomputed projection), so the
    decode equals the oracle's decode with W^R = I."""
    x = tiny(B=3, Hq=16, Hkv=4, D=128, P=16, lens=(1, 300, 1000))
    k = _kernel_or_skip(kname, x)
    g = to_dev(x)
    sh = shape_of(x)
    out = torch.full((3, 16, 128), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, num_splits)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_attention_ex(sh, g["q"], None, g["v_cache"], g["block_table"], g["seq_lens"],
                              kl.decode_options(num_splits, k), out, kl.KL_FP32, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    eye = np.broadcast_to(np.eye(128, dtype=np.float32)[None], (4, 128, 128))
    w_eye = bf16_bits(torch.from_numpy(eye.copy()).to(torch.bfloat16))
    want = oracle.decode(bf16_bits(x["q"]), w_eye, bf16_bits(x["v_cache"]),
                         x["block_table"].numpy(), x["seq_lens"].numpy(),
                         scale=_gpu.default_scale(x))
    assert_parity(out.cpu().numpy(), want, f"composed query {kname} S={num_splits}")


def test_composed_query_fused_step_appends_and_decodes():
    x = tiny(B=2, Hq=32, Hkv=8, D=128, P=32, lens=(700, 64))
    if not _tc_available(x):
        pytest.skip("tensor-core kernel does not support this geometry")
    g = to_dev(x)
    sh = shape_of(x)
    out = torch.empty(2, 32, 128, dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    ws = torch.zeros(max(256, kl.kl_decode_workspace_size(sh, 2)), dtype=torch.uint8,
                     device=_gpu.dev())
    kl.kl_decode_step(sh, g["q"], None, g["v_new"], g["positions"], g["v_cache"],
                      g["block_table"], g["seq_lens"], kl.decode_options(2), out, kl.KL_FP32, ws,
                      err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    cache = oracle.append(bf16_bits(x["v_cache"]), bf16_bits(x["v_new"]),
                          x["block_table"].numpy(), x["positions"].numpy())
    eye = np.broadcast_to(np.eye(128, dtype=np.float32)[None], (8, 128, 128))
    w_eye = bf16_bits(torch.from_numpy(eye.copy()).to(torch.bfloat16))
    want = oracle.decode(bf16_bits(x["q"]), w_eye, cache, x["block_table"].numpy(),
                         x["seq_lens"].numpy(), scale=_gpu.default_scale(x))
    assert_parity(out.cpu().numpy(), want, "composed query, fused step")


# ------------------------------------------------------------------ split-state outputs -----

@pytest.mark.parametrize("splits", [3, 64])
@pytest.mark.parametrize("G", [4, 8])
def test_split_states_match_oracle_partial_states(splits, G):
    """The split states the caller asks for (partial_o / partial_ml): every split's normalized
    output, largest score and exponent sum against the oracle's states of the same token
    ranges, then their merge by kl_combine. At 64 splits of a 2-sequence, 8-value-head batch
    one CTA runs several consecutive splits and writes a state at each split boundary."""
    x = tiny(B=2, Hq=8 * G, Hkv=8, D=128, P=16, lens=(2000, 4096), seed=23)
    k = _kernel_or_skip("tensor", x)
    g = to_dev(x)
    sh = shape_of(x)
    B, Hq, D = x["q"].shape
    S = kl.kl_decode_num_splits(sh, splits)
    lmax = x["block_table"].shape[1] * 16
    chunk = -(-(-(-lmax // S)) // 128) * 128            # ceil(lmax / S), rounded up to 128
    po = torch.full((B, Hq, S, D), float("nan"), dtype=torch.float32, device=_gpu.dev())
    pml = torch.full((B, Hq, S, 2), float("nan"), dtype=torch.float32, device=_gpu.dev())
    err = torch.zeros(1, dtype=torch.int32, device=_gpu.dev())
    kl.kl_decode_attention_ex(sh, g["q"], g["w_r"], g["v_cache"], g["block_table"],
                              g["seq_lens"], kl.decode_options(splits, k, po, pml), None,
                              kl.KL_FP32, None, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    want_o, want_ml = oracle.decode_partial(bf16_bits(x["q"]), bf16_bits(x["w_r"]),
                                            bf16_bits(x["v_cache"]), x["block_table"].numpy(),
                                            x["seq_lens"].numpy(), scale=_gpu.default_scale(x),
                                            chunk=chunk, num_splits=S)
    got_o, got_ml = po.cpu().numpy().astype(np.float64), pml.cpu().numpy().astype(np.float64)
    full = want_ml[..., 1] > 0
    assert np.array_equal(got_ml[..., 1] > 0, full), "empty splits differ"
    assert np.all(np.isneginf(got_ml[..., 0][~full])) and np.all(got_o[~full] == 0.0)
    assert_parity(got_o[full], want_o[full], f"split states S={S}")
    m_g, m_w = got_ml[..., 0][full], want_ml[..., 0][full]
    assert np.all(np.abs(m_g - m_w) <= 1e-3 + 1e-4 * np.abs(m_w)), "largest scores differ"
    l_g, l_w = got_ml[..., 1][full], want_ml[..., 1][full]
    assert np.all(np.abs(l_g - l_w) <= 1e-3 * l_w), "exponent sums differ"
    out = torch.empty(B, Hq, D, dtype=torch.float32, device=_gpu.dev())
    kl.kl_combine(sh, po, pml, S, out, kl.KL_FP32)
    torch.cuda.synchronize()
    assert_parity(out.cpu().numpy(), oracle_decode(x, _gpu.default_scale(x)), "combined states")
