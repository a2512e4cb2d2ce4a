"""GB300-native decode (and chunked prefill) of Keyless Attention over a paged Value-Only Cache.

The compute lives in ``libkeyless.so`` (hand-written CUDA for sm_103a behind the C ABI of
``include/keyless.h``); this package holds its build script, a ctypes binding with the same
function names, and the seeded input generators. PyTorch is used for device memory and
streams only.
"""
from .builder import build  # noqa: F401
from ._lib import (  # noqa: F401
    KL_BF16, KL_FP32, KL_KERNEL_AUTO, KL_KERNEL_SIMT, KL_KERNEL_TENSOR, KL_OK,
    KL_ERR_CUDA, KL_ERR_INVALID_ARG, KL_ERR_UNSUPPORTED, KL_ERR_WORKSPACE,
    KL_FLAG_BAD_LENGTH, KL_FLAG_BAD_PAGE, KL_FLAG_BAD_POSITION, KL_FLAG_RANGE, KL_FLAG_TIMEOUT,
    KLError, decode_options, kl_append_v, kl_combine, kl_decode_attention, kl_decode_attention_ex,
    kl_decode_attention_noalloc, kl_decode_kernel_available, kl_decode_step, KL_NOALLOC_SCRATCH_BYTES,
    kl_decode_num_splits, kl_decode_options, kl_decode_workspace_size, kl_route_query,
    kl_shape, kl_standard_decode, kl_status_string, load, make_shape,
    kl_append_v_chunk, kl_prefill_attention,
    kl_latent_shape, make_latent_shape, kl_latent_workspace_size, kl_latent_decode,
    kl_latent_decode_step,
    kl_append_v_fp8, kl_decode_attention_fp8, kl_decode_step_fp8, kl_quantize_cache_fp8,
    kl_set_wait_timeout_ns,
)
