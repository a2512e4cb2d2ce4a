"""fp64 CPU oracle for Keyless Attention decode over a paged Value-Only Cache.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg
of ``bench.py`` import this package. The product path (the CUDA library under
``paper_2606_21848_gb300`` and its binding) never imports it, and the two share no code.

Two independent formulations live here:

* ``keyless_oracle.c`` (loaded through ctypes) -- the paged definition, written out in plain
  C with fp64 arithmetic: routing projection q_r = q W^R (Eq. 2, Section 2.2), scores
  s_i = scale * <q_r, v_i>, softmax weights alpha_{n+1,i} and output O_{n+1} = sum alpha v_i
  (Section 3), plus the split-state merge, the cache append and, for the K+V comparison,
  standard attention (Eq. 1).
  The prefill of a chunk of new tokens (Eq. 3 with a causal mask), the chunk append, the
  decode over a latent value-only cache (Section 3) and over an FP8 (E4M3, per-row scale) value
  cache use the same per-row attention.
* ``dense.py`` -- a NumPy brute force that first un-pages the cache with its own code and then
  evaluates the same formulas on dense arrays; it is used for tiny inputs only.

All bf16 inputs are passed as uint16 bit patterns and widened exactly.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "keyless_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libkeyless_oracle.so")

_lib = None
_openmp = None


def build(force: bool = False) -> str:
    """Compile the C oracle with gcc (OpenMP when the toolchain has it). Returns the .so path."""
    global _openmp
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    base = ["gcc", "-O2", "-fPIC", "-shared", "-std=c11", _SRC, "-o", _LIB_PATH + ".tmp", "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
        _openmp = True
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
        _openmp = False
    os.replace(_LIB_PATH + ".tmp", _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        i, d, p = ctypes.c_int, ctypes.c_double, ctypes.c_void_p
        _lib.ko_route.argtypes = [i, i, i, i, i, p, p, p]
        _lib.ko_decode.argtypes = [i, i, i, i, i, i, i, i, d, p, p, p, p, p, i, p, p]
        _lib.ko_standard_decode.argtypes = [i, i, i, i, i, i, i, d, p, p, p, p, p, i, p, p]
        _lib.ko_attention_weights.argtypes = [i, i, i, i, i, i, i, i, d, p, p, p, p, p, i, i, p]
        _lib.ko_decode_partial.argtypes = [i, i, i, i, i, i, i, i, d, p, p, p, p, p, i, i, p, p]
        _lib.ko_combine.argtypes = [i, i, i, i, p, p, p]
        _lib.ko_append.argtypes = [i, i, i, i, i, i, p, p, p, p]
        _lib.ko_prefill.argtypes = [i, i, i, i, i, i, i, i, d, p, p, p, p, p, p, i, p, p]
        _lib.ko_append_chunk.argtypes = [i, i, i, i, i, i, p, p, p, p, p]
        _lib.ko_latent_decode.argtypes = [i, i, i, i, i, i, i, i, i, d, p, p, p, p, p, p, i, p, p]
        _lib.ko_quantize_rows.argtypes = [i, i, p, p, p]
        _lib.ko_append_fp8.argtypes = [i, i, i, i, i, i, p, p, p, p, p]
        _lib.ko_decode_fp8.argtypes = [i, i, i, i, i, i, i, i, d, p, p, p, p, p, p, i, p, p]
        for f in ("ko_route", "ko_decode", "ko_standard_decode", "ko_attention_weights",
                  "ko_decode_partial", "ko_combine", "ko_append", "ko_prefill",
                  "ko_append_chunk", "ko_latent_decode", "ko_quantize_rows", "ko_append_fp8",
                  "ko_decode_fp8"):
            getattr(_lib, f).restype = ctypes.c_int
        _lib.ko_e4m3_from_f32.argtypes = [ctypes.c_float]
        _lib.ko_e4m3_from_f32.restype = ctypes.c_uint8
        _lib.ko_e4m3_value.argtypes = [ctypes.c_uint8]
        _lib.ko_e4m3_value.restype = ctypes.c_double
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a: np.ndarray, dtype) -> np.ndarray:
    a = np.ascontiguousarray(a)
    if a.dtype != dtype:
        raise TypeError(f"expected {np.dtype(dtype)}, got {a.dtype}")
    return a


def threads() -> int:
    """Threads the oracle's OpenMP loops use (1 when built without OpenMP)."""
    build()
    if _openmp is False:
        return 1
    return int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))


def _check(rc: int, what: str):
    if rc != 0:
        raise ValueError(f"oracle {what}: an index, position or length is out of range")


def route(q, w_r, num_kv_heads: int, wr_per_query_head: bool = False) -> np.ndarray:
    """q_r[b, h] = q[b, h] @ W^R[w(h)] in fp64; q [B, Hq, D] and w_r [Hw, D, D] as bf16 bits."""
    q = _c(q, np.uint16)
    w_r = _c(w_r, np.uint16)
    B, Hq, D = q.shape
    out = np.zeros((B, Hq, D), np.float64)
    _check(_load().ko_route(B, Hq, num_kv_heads, D, int(wr_per_query_head), _ptr(q), _ptr(w_r),
                            _ptr(out)), "route")
    return out


def decode(q, w_r, v_cache, block_table, seq_lens, *, scale: float,
           wr_per_query_head: bool = False, heads=None) -> np.ndarray:
    """Keyless decode (Section 3). Returns [B, Hq, D] fp64, or [len(heads), D] for (b, h) pairs."""
    q, w_r, v_cache = _c(q, np.uint16), _c(w_r, np.uint16), _c(v_cache, np.uint16)
    bt, sl = _c(block_table, np.int32), _c(seq_lens, np.int32)
    B, Hq, D = q.shape
    num_pages, Hkv, P, _ = v_cache.shape
    sel = None if heads is None else _c(np.asarray(heads, np.int32).reshape(-1, 2), np.int32)
    out = np.zeros(((B * Hq) if sel is None else len(sel), D), np.float64)
    rc = _load().ko_decode(B, Hq, Hkv, D, P, num_pages, bt.shape[1], int(wr_per_query_head),
                           float(scale), _ptr(q), _ptr(w_r), _ptr(v_cache), _ptr(bt), _ptr(sl),
                           0 if sel is None else len(sel), _ptr(sel), _ptr(out))
    _check(rc, "decode")
    return out.reshape(B, Hq, D) if sel is None else out


def standard_decode(q, k_cache, v_cache, block_table, seq_lens, *, scale: float,
                    heads=None) -> np.ndarray:
    """Standard attention decode over paged K and V caches (Eq. 1), the comparison path."""
    q, k_cache, v_cache = _c(q, np.uint16), _c(k_cache, np.uint16), _c(v_cache, np.uint16)
    bt, sl = _c(block_table, np.int32), _c(seq_lens, np.int32)
    B, Hq, D = q.shape
    num_pages, Hkv, P, _ = v_cache.shape
    sel = None if heads is None else _c(np.asarray(heads, np.int32).reshape(-1, 2), np.int32)
    out = np.zeros(((B * Hq) if sel is None else len(sel), D), np.float64)
    rc = _load().ko_standard_decode(B, Hq, Hkv, D, P, num_pages, bt.shape[1], float(scale),
                                    _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(bt), _ptr(sl),
                                    0 if sel is None else len(sel), _ptr(sel), _ptr(out))
    _check(rc, "standard_decode")
    return out.reshape(B, Hq, D) if sel is None else out


def attention_weights(q, w_r, v_cache, block_table, seq_lens, b: int, h: int, *, scale: float,
                      wr_per_query_head: bool = False) -> np.ndarray:
    """alpha_{n+1, i} for one (b, h), i over the L_b cached rows (Section 3)."""
    q, w_r, v_cache = _c(q, np.uint16), _c(w_r, np.uint16), _c(v_cache, np.uint16)
    bt, sl = _c(block_table, np.int32), _c(seq_lens, np.int32)
    B, Hq, D = q.shape
    num_pages, Hkv, P, _ = v_cache.shape
    alpha = np.zeros(max(int(sl[b]), 1), np.float64)
    rc = _load().ko_attention_weights(B, Hq, Hkv, D, P, num_pages, bt.shape[1],
                                      int(wr_per_query_head), float(scale), _ptr(q), _ptr(w_r),
                                      _ptr(v_cache), _ptr(bt), _ptr(sl), b, h, _ptr(alpha))
    _check(rc, "attention_weights")
    return alpha[: int(sl[b])]


def decode_partial(q, w_r, v_cache, block_table, seq_lens, *, scale: float, chunk: int,
                   num_splits: int, wr_per_query_head: bool = False):
    """Split states (o, (m, l)) for splits [s*chunk, (s+1)*chunk): [B,Hq,S,D] and [B,Hq,S,2]."""
    q, w_r, v_cache = _c(q, np.uint16), _c(w_r, np.uint16), _c(v_cache, np.uint16)
    bt, sl = _c(block_table, np.int32), _c(seq_lens, np.int32)
    B, Hq, D = q.shape
    num_pages, Hkv, P, _ = v_cache.shape
    po = np.zeros((B, Hq, num_splits, D), np.float64)
    pml = np.zeros((B, Hq, num_splits, 2), np.float64)
    rc = _load().ko_decode_partial(B, Hq, Hkv, D, P, num_pages, bt.shape[1],
                                   int(wr_per_query_head), float(scale), _ptr(q), _ptr(w_r),
                                   _ptr(v_cache), _ptr(bt), _ptr(sl), chunk, num_splits,
                                   _ptr(po), _ptr(pml))
    _check(rc, "decode_partial")
    return po, pml


def combine(part_o, part_ml) -> np.ndarray:
    """Merge split states [B,Hq,S,D] + [B,Hq,S,2] (m, l) into one output [B,Hq,D] (fp64)."""
    po = np.ascontiguousarray(part_o, dtype=np.float64)
    pml = np.ascontiguousarray(part_ml, dtype=np.float64)
    B, Hq, S, D = po.shape
    out = np.zeros((B, Hq, D), np.float64)
    _check(_load().ko_combine(B, Hq, D, S, _ptr(po), _ptr(pml), _ptr(out)), "combine")
    return out


def append(v_cache, v_new, block_table, positions) -> np.ndarray:
    """Return a copy of the cache with v_new[b, g] written at row positions[b] (bit copy)."""
    cache = np.array(_c(v_cache, np.uint16), copy=True)
    v_new = _c(v_new, np.uint16)
    bt, pos = _c(block_table, np.int32), _c(positions, np.int32)
    num_pages, Hkv, P, D = cache.shape
    B = v_new.shape[0]
    rc = _load().ko_append(B, Hkv, D, P, num_pages, bt.shape[1], _ptr(v_new), _ptr(bt),
                           _ptr(pos), _ptr(cache))
    _check(rc, "append")
    return cache


def prefill(q, w_r, v_cache, block_table, seq_lens, cu_q, *, scale: float,
            wr_per_query_head: bool = False, rows=None) -> np.ndarray:
    """Keyless prefill of chunks under the causal mask: [T, Hq, D] fp64, or [len(rows), D].

    q is [T, Hq, D] (bf16 bits), the rows of sequence b being cu_q[b]..cu_q[b+1]-1; the chunk
    is the last cu_q[b+1]-cu_q[b] of the seq_lens[b] cached rows. ``rows`` selects (r, h) pairs.
    """
    q, w_r, v_cache = _c(q, np.uint16), _c(w_r, np.uint16), _c(v_cache, np.uint16)
    bt, sl, cu = _c(block_table, np.int32), _c(seq_lens, np.int32), _c(cu_q, np.int32)
    T, Hq, D = q.shape
    num_pages, Hkv, P, _ = v_cache.shape
    B = len(sl)
    if len(cu) != B + 1 or int(cu[-1]) != T:
        raise ValueError("cu_q must have B + 1 entries ending at the number of query rows")
    sel = None if rows is None else _c(np.asarray(rows, np.int32).reshape(-1, 2), np.int32)
    out = np.zeros(((T * Hq) if sel is None else len(sel), D), np.float64)
    rc = _load().ko_prefill(B, Hq, Hkv, D, P, num_pages, bt.shape[1], int(wr_per_query_head),
                            float(scale), _ptr(q), _ptr(w_r), _ptr(v_cache), _ptr(bt), _ptr(sl),
                            _ptr(cu), 0 if sel is None else len(sel), _ptr(sel), _ptr(out))
    _check(rc, "prefill")
    return out.reshape(T, Hq, D) if sel is None else out


def append_chunk(v_cache, v_new, block_table, seq_lens, cu_q) -> np.ndarray:
    """Copy of the cache with the rows of each chunk written at positions L_b - n_b .. L_b - 1."""
    cache = np.array(_c(v_cache, np.uint16), copy=True)
    v_new = _c(v_new, np.uint16)
    bt, sl, cu = _c(block_table, np.int32), _c(seq_lens, np.int32), _c(cu_q, np.int32)
    num_pages, Hkv, P, D = cache.shape
    rc = _load().ko_append_chunk(len(sl), Hkv, D, P, num_pages, bt.shape[1], _ptr(v_new),
                                 _ptr(bt), _ptr(sl), _ptr(cu), _ptr(cache))
    _check(rc, "append_chunk")
    return cache


def latent_decode(q, w_r, w_post, v_lat, block_table, seq_lens, *, scale: float,
                  wr_per_query_head: bool = False, heads=None) -> np.ndarray:
    """Decode over a latent value-only cache (Section 3): absorbed query q* = (q W^R) W_post^T,
    softmax(scale q* V*^T) V* W_post. q [B, Hq, D], w_post [Hq, r, D], v_lat [pages, Hl, P, r]
    (bf16 bits). Returns [B, Hq, D] fp64, or [len(heads), D] for (b, h) pairs."""
    q, w_r, w_post = _c(q, np.uint16), _c(w_r, np.uint16), _c(w_post, np.uint16)
    v_lat = _c(v_lat, np.uint16)
    bt, sl = _c(block_table, np.int32), _c(seq_lens, np.int32)
    B, Hq, D = q.shape
    num_pages, Hl, P, r = v_lat.shape
    if w_post.shape != (Hq, r, D):
        raise ValueError("w_post must be [Hq, r, D]")
    sel = None if heads is None else _c(np.asarray(heads, np.int32).reshape(-1, 2), np.int32)
    out = np.zeros(((B * Hq) if sel is None else len(sel), D), np.float64)
    rc = _load().ko_latent_decode(B, Hq, Hl, D, r, P, num_pages, bt.shape[1],
                                  int(wr_per_query_head), float(scale), _ptr(q), _ptr(w_r),
                                  _ptr(w_post), _ptr(v_lat), _ptr(bt), _ptr(sl),
                                  0 if sel is None else len(sel), _ptr(sel), _ptr(out))
    _check(rc, "latent_decode")
    return out.reshape(B, Hq, D) if sel is None else out


# ----------------------------------------------------------------- FP8 value cache ----------

def e4m3_value(codes) -> np.ndarray:
    """Values of OCP FP8 E4M3 codes (uint8) as float64 (NaN for the NaN codes)."""
    lib = _load()
    c = np.asarray(codes, np.uint8)
    return np.array([lib.ko_e4m3_value(int(x)) for x in c.ravel()], np.float64).reshape(c.shape)


def e4m3_from_f32(x) -> np.ndarray:
    """Nearest E4M3 codes of float32 values (ties to even mantissa, saturating at 448)."""
    lib = _load()
    a = np.asarray(x, np.float32)
    return np.array([lib.ko_e4m3_from_f32(float(v)) for v in a.ravel()], np.uint8).reshape(a.shape)


def quantize_rows(v_bits) -> tuple[np.ndarray, np.ndarray]:
    """Per-row FP8 quantization of bf16 rows [..., D]: codes uint8 [..., D], scales float32 [...]."""
    v = _c(v_bits, np.uint16)
    D = v.shape[-1]
    n = v.size // D
    codes = np.zeros(v.shape, np.uint8)
    scales = np.zeros(v.shape[:-1], np.float32)
    _load().ko_quantize_rows(n, D, _ptr(v), _ptr(codes), _ptr(scales))
    return codes, scales


def append_fp8(codes, scales, v_new, block_table, positions):
    """Copies of the FP8 cache (codes [pages, Hkv, P, D], scales [pages, Hkv, P]) with v_new[b]
    quantized into row positions[b]."""
    codes = np.array(_c(codes, np.uint8), copy=True)
    scales = np.array(_c(scales, np.float32), copy=True)
    v_new = _c(v_new, np.uint16)
    bt, pos = _c(block_table, np.int32), _c(positions, np.int32)
    num_pages, Hkv, P, D = codes.shape
    rc = _load().ko_append_fp8(v_new.shape[0], Hkv, D, P, num_pages, bt.shape[1], _ptr(v_new),
                               _ptr(bt), _ptr(pos), _ptr(codes), _ptr(scales))
    _check(rc, "append_fp8")
    return codes, scales


def decode_fp8(q, w_r, codes, scales, block_table, seq_lens, *, scale: float,
               wr_per_query_head: bool = False, heads=None) -> np.ndarray:
    """Keyless decode over the FP8 cache (values scale * e4m3(code)); [B, Hq, D] fp64."""
    q, w_r = _c(q, np.uint16), _c(w_r, np.uint16)
    codes, scales = _c(codes, np.uint8), _c(scales, np.float32)
    bt, sl = _c(block_table, np.int32), _c(seq_lens, np.int32)
    B, Hq, D = q.shape
    num_pages, Hkv, P, _ = codes.shape
    sel = None if heads is None else _c(np.asarray(heads, np.int32).reshape(-1, 2), np.int32)
    out = np.zeros(((B * Hq) if sel is None else len(sel), D), np.float64)
    rc = _load().ko_decode_fp8(B, Hq, Hkv, D, P, num_pages, bt.shape[1], int(wr_per_query_head),
                               float(scale), _ptr(q), _ptr(w_r), _ptr(codes), _ptr(scales),
                               _ptr(bt), _ptr(sl), 0 if sel is None else len(sel), _ptr(sel),
                               _ptr(out))
    _check(rc, "decode_fp8")
    return out.reshape(B, Hq, D) if sel is None else out
