"""ctypes binding of libkeyless (include/keyless.h): argument marshalling only.

Every function has the C name and the C argument order; tensors are passed as torch CUDA
tensors (or raw device addresses as ints) and the stream defaults to torch's current stream.
A non-OK status raises :class:`KLError`. There is no fallback: if the library has not been
built, :func:`load` raises.
"""
from __future__ import annotations

import ctypes
import os
import re

from . import builder as _build

KL_OK, KL_ERR_INVALID_ARG, KL_ERR_UNSUPPORTED, KL_ERR_WORKSPACE, KL_ERR_CUDA = range(5)
KL_BF16, KL_FP32 = 0, 1
KL_KERNEL_AUTO, KL_KERNEL_TENSOR, KL_KERNEL_SIMT = 0, 1, 2
KL_FLAG_BAD_PAGE, KL_FLAG_BAD_POSITION, KL_FLAG_BAD_LENGTH, KL_FLAG_TIMEOUT, KL_FLAG_RANGE = 1, 2, 4, 8, 16
KL_NOALLOC_SCRATCH_BYTES = 32 * 1024 * 1024

HEADER = os.path.join(_build.INCLUDE, "keyless.h")


class KLError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


class kl_shape(ctypes.Structure):
    _fields_ = [("num_seqs", ctypes.c_int32), ("num_q_heads", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("num_pages", ctypes.c_int32),
                ("max_pages_per_seq", ctypes.c_int32), ("wr_per_query_head", ctypes.c_int32),
                ("scale", ctypes.c_float)]


class kl_latent_shape(ctypes.Structure):
    _fields_ = [("num_seqs", ctypes.c_int32), ("num_q_heads", ctypes.c_int32),
                ("num_latent_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("latent_dim", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("num_pages", ctypes.c_int32), ("max_pages_per_seq", ctypes.c_int32),
                ("wr_per_query_head", ctypes.c_int32), ("scale", ctypes.c_float)]


class kl_decode_options(ctypes.Structure):
    _fields_ = [("num_splits", ctypes.c_int32), ("kernel", ctypes.c_int32),
                ("partial_o", ctypes.c_void_p), ("partial_ml", ctypes.c_void_p)]


def decode_options(num_splits=0, kernel=KL_KERNEL_AUTO, partial_o=None, partial_ml=None):
    """kl_decode_options; partial_o / partial_ml are tensors (or addresses) for split states."""
    addr = lambda t: None if t is None else (t if isinstance(t, int) else t.data_ptr())
    return kl_decode_options(num_splits, kernel, addr(partial_o), addr(partial_ml))


_lib = None


def load() -> ctypes.CDLL:
    """Load the built library (raises if it is missing; run build() first)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_build.LIB):
        raise RuntimeError(f"libkeyless is not built ({_build.LIB} missing); call build() first")
    lib = ctypes.CDLL(_build.LIB)
    P, I32, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    SH = ctypes.POINTER(kl_shape)
    OP = ctypes.POINTER(kl_decode_options)
    LS = ctypes.POINTER(kl_latent_shape)
    sig = {
        "kl_route_query": ([SH, P, P, P, P], I32),
        "kl_append_v": ([SH, P, P, P, P, P, P], I32),
        "kl_decode_workspace_size": ([SH, I32], SZ),
        "kl_decode_num_splits": ([SH, I32], I32),
        "kl_decode_attention": ([SH, P, P, P, P, P, I32, P, I32, P, SZ, P, P], I32),
        "kl_decode_attention_ex": ([SH, P, P, P, P, P, OP, P, I32, P, SZ, P, P], I32),
        "kl_combine": ([SH, P, P, I32, P, I32, P], I32),
        "kl_standard_decode": ([SH, P, P, P, P, P, OP, P, I32, P, SZ, P, P], I32),
        "kl_decode_step": ([SH, P, P, P, P, P, P, P, OP, P, I32, P, SZ, P, P], I32),
        "kl_decode_attention_noalloc": ([SH, P, P, P, P, P, I32, P, I32, P, P], I32),
        "kl_decode_kernel_available": ([SH, I32, I32], I32),
        "kl_append_v_chunk": ([SH, P, P, P, P, I32, I32, P, P, P], I32),
        "kl_append_v_fp8": ([SH, P, P, P, P, P, P, P], I32),
        "kl_quantize_cache_fp8": ([SH, P, P, P, P], I32),
        "kl_decode_attention_fp8": ([SH, P, P, P, P, P, P, I32, P, I32, P, SZ, P, P], I32),
        "kl_decode_step_fp8": ([SH, P, P, P, P, P, P, P, P, I32, P, I32, P, SZ, P, P], I32),
        "kl_latent_workspace_size": ([LS, I32], SZ),
        "kl_latent_decode": ([LS, P, P, P, P, P, P, I32, P, I32, P, SZ, P, P], I32),
        "kl_latent_decode_step": ([LS, P, P, P, P, P, P, P, P, I32, P, I32, P, SZ, P, P], I32),
        "kl_prefill_attention": ([SH, P, P, P, P, P, P, I32, I32, P, I32, P, P], I32),
        "kl_set_wait_timeout_ns": ([ctypes.c_uint64], ctypes.c_uint64),
        "kl_status_string": ([I32], ctypes.c_char_p),
    }
    for name, (args, res) in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    _lib = lib
    return lib


def declared_symbols() -> list[str]:
    """Names of the functions include/keyless.h declares."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\s\*]*?\b(kl_\w+)\s*\(", text, re.M)))


def status_string(status: int) -> str:
    try:
        return load().kl_status_string(status).decode()
    except Exception:  # the library could not be loaded
        return "unknown"


def _p(x):
    if x is None:
        return None
    if isinstance(x, int):
        return ctypes.c_void_p(x)
    return ctypes.c_void_p(x.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _nbytes(t) -> int:
    return 0 if t is None else t.numel() * t.element_size()


def _check(status: int, where: str):
    if status != KL_OK:
        raise KLError(status, where)


def make_shape(num_seqs, num_q_heads, num_kv_heads, head_dim, page_size, num_pages,
               max_pages_per_seq, wr_per_query_head=False, scale=0.0) -> kl_shape:
    return kl_shape(num_seqs, num_q_heads, num_kv_heads, head_dim, page_size, num_pages,
                    max_pages_per_seq, int(bool(wr_per_query_head)), float(scale))


def kl_route_query(shape, q, w_r, q_r, stream=None):
    _check(load().kl_route_query(ctypes.byref(shape), _p(q), _p(w_r), _p(q_r), _stream(stream)),
           "kl_route_query")


def kl_append_v(shape, v_new, block_table, positions, v_cache, err=None, stream=None):
    _check(load().kl_append_v(ctypes.byref(shape), _p(v_new), _p(block_table), _p(positions),
                              _p(v_cache), _p(err), _stream(stream)), "kl_append_v")


def kl_decode_workspace_size(shape, num_splits=0) -> int:
    return int(load().kl_decode_workspace_size(ctypes.byref(shape), num_splits))


def kl_decode_num_splits(shape, num_splits=0) -> int:
    return int(load().kl_decode_num_splits(ctypes.byref(shape), num_splits))


def kl_decode_attention(shape, q, w_r, v_cache, block_table, seq_lens, num_splits, out,
                        out_dtype, workspace, err=None, stream=None):
    _check(load().kl_decode_attention(ctypes.byref(shape), _p(q), _p(w_r), _p(v_cache),
                                      _p(block_table), _p(seq_lens), num_splits, _p(out),
                                      out_dtype, _p(workspace), _nbytes(workspace), _p(err),
                                      _stream(stream)), "kl_decode_attention")


def kl_decode_attention_ex(shape, q, w_r, v_cache, block_table, seq_lens, opts, out,
                           out_dtype, workspace, err=None, stream=None):
    _check(load().kl_decode_attention_ex(ctypes.byref(shape), _p(q), _p(w_r), _p(v_cache),
                                         _p(block_table), _p(seq_lens),
                                         None if opts is None else ctypes.byref(opts), _p(out),
                                         out_dtype, _p(workspace), _nbytes(workspace), _p(err),
                                         _stream(stream)), "kl_decode_attention_ex")


def kl_decode_step(shape, q, w_r, v_new, positions, v_cache, block_table, seq_lens, opts, out,
                   out_dtype, workspace, err=None, stream=None):
    """Append of the current token's rows fused with the keyless decode (one pass)."""
    _check(load().kl_decode_step(ctypes.byref(shape), _p(q), _p(w_r), _p(v_new), _p(positions),
                                 _p(v_cache), _p(block_table), _p(seq_lens),
                                 None if opts is None else ctypes.byref(opts), _p(out),
                                 out_dtype, _p(workspace), _nbytes(workspace), _p(err),
                                 _stream(stream)), "kl_decode_step")


def kl_combine(shape, partial_o, partial_ml, num_splits, out, out_dtype, stream=None):
    _check(load().kl_combine(ctypes.byref(shape), _p(partial_o), _p(partial_ml), num_splits,
                             _p(out), out_dtype, _stream(stream)), "kl_combine")


def kl_standard_decode(shape, q, k_cache, v_cache, block_table, seq_lens, opts, out, out_dtype,
                       workspace, err=None, stream=None):
    _check(load().kl_standard_decode(ctypes.byref(shape), _p(q), _p(k_cache), _p(v_cache),
                                     _p(block_table), _p(seq_lens),
                                     None if opts is None else ctypes.byref(opts), _p(out),
                                     out_dtype, _p(workspace), _nbytes(workspace), _p(err),
                                     _stream(stream)), "kl_standard_decode")


def kl_decode_attention_noalloc(shape, q, w_r, v_cache, block_table, seq_lens, num_splits, out,
                                out_dtype, err=None, stream=None):
    """The decode with its split states in the library's fixed device scratch (no workspace)."""
    _check(load().kl_decode_attention_noalloc(ctypes.byref(shape), _p(q), _p(w_r), _p(v_cache),
                                              _p(block_table), _p(seq_lens), num_splits, _p(out),
                                              out_dtype, _p(err), _stream(stream)),
           "kl_decode_attention_noalloc")


def kl_append_v_chunk(shape, v_new, block_table, seq_lens, cu_q_lens, total_q, max_q_len, v_cache,
                      err=None, stream=None):
    _check(load().kl_append_v_chunk(ctypes.byref(shape), _p(v_new), _p(block_table), _p(seq_lens),
                                    _p(cu_q_lens), total_q, max_q_len, _p(v_cache), _p(err),
                                    _stream(stream)), "kl_append_v_chunk")


def kl_prefill_attention(shape, q, w_r, v_cache, block_table, seq_lens, cu_q_lens, total_q,
                         max_q_len, out, out_dtype, err=None, stream=None):
    _check(load().kl_prefill_attention(ctypes.byref(shape), _p(q), _p(w_r), _p(v_cache),
                                       _p(block_table), _p(seq_lens), _p(cu_q_lens), total_q,
                                       max_q_len, _p(out), out_dtype, _p(err), _stream(stream)),
           "kl_prefill_attention")


def kl_append_v_fp8(shape, v_new, block_table, positions, v_codes, v_scales, err=None,
                    stream=None):
    _check(load().kl_append_v_fp8(ctypes.byref(shape), _p(v_new), _p(block_table), _p(positions),
                                  _p(v_codes), _p(v_scales), _p(err), _stream(stream)),
           "kl_append_v_fp8")


def kl_quantize_cache_fp8(shape, v_cache, v_codes, v_scales, stream=None):
    _check(load().kl_quantize_cache_fp8(ctypes.byref(shape), _p(v_cache), _p(v_codes),
                                        _p(v_scales), _stream(stream)), "kl_quantize_cache_fp8")


def kl_decode_attention_fp8(shape, q, w_r, v_codes, v_scales, block_table, seq_lens, num_splits,
                            out, out_dtype, workspace, err=None, stream=None):
    _check(load().kl_decode_attention_fp8(ctypes.byref(shape), _p(q), _p(w_r), _p(v_codes),
                                          _p(v_scales), _p(block_table), _p(seq_lens), num_splits,
                                          _p(out), out_dtype, _p(workspace), _nbytes(workspace),
                                          _p(err), _stream(stream)), "kl_decode_attention_fp8")


def kl_decode_step_fp8(shape, q, w_r, v_new, positions, v_codes, v_scales, block_table, seq_lens,
                       num_splits, out, out_dtype, workspace, err=None, stream=None):
    _check(load().kl_decode_step_fp8(ctypes.byref(shape), _p(q), _p(w_r), _p(v_new), _p(positions),
                                     _p(v_codes), _p(v_scales), _p(block_table), _p(seq_lens),
                                     num_splits, _p(out), out_dtype, _p(workspace),
                                     _nbytes(workspace), _p(err), _stream(stream)),
           "kl_decode_step_fp8")


def make_latent_shape(num_seqs, num_q_heads, num_latent_heads, head_dim, latent_dim, page_size,
                      num_pages, max_pages_per_seq, wr_per_query_head=False, scale=0.0):
    return kl_latent_shape(num_seqs, num_q_heads, num_latent_heads, head_dim, latent_dim,
                           page_size, num_pages, max_pages_per_seq, int(bool(wr_per_query_head)),
                           float(scale))


def kl_latent_workspace_size(shape, num_splits=0) -> int:
    return int(load().kl_latent_workspace_size(ctypes.byref(shape), num_splits))


def kl_latent_decode(shape, q, w_r, w_post, v_lat, block_table, seq_lens, num_splits, out,
                     out_dtype, workspace, err=None, stream=None):
    _check(load().kl_latent_decode(ctypes.byref(shape), _p(q), _p(w_r), _p(w_post), _p(v_lat),
                                   _p(block_table), _p(seq_lens), num_splits, _p(out), out_dtype,
                                   _p(workspace), _nbytes(workspace), _p(err), _stream(stream)),
           "kl_latent_decode")


def kl_latent_decode_step(shape, q, w_r, w_post, v_new, positions, v_lat, block_table, seq_lens,
                          num_splits, out, out_dtype, workspace, err=None, stream=None):
    _check(load().kl_latent_decode_step(ctypes.byref(shape), _p(q), _p(w_r), _p(w_post), _p(v_new),
                                        _p(positions), _p(v_lat), _p(block_table), _p(seq_lens),
                                        num_splits, _p(out), out_dtype, _p(workspace),
                                        _nbytes(workspace), _p(err), _stream(stream)),
           "kl_latent_decode_step")


def kl_decode_kernel_available(shape, kernel, standard=False) -> bool:
    return bool(load().kl_decode_kernel_available(ctypes.byref(shape), kernel, int(standard)))


def kl_set_wait_timeout_ns(ns: int) -> int:
    """Set the decodes' pipeline-wait limit (ns; 0 = the default); returns the previous one."""
    return int(load().kl_set_wait_timeout_ns(int(ns)))


def kl_status_string(status: int) -> str:
    return status_string(status)
