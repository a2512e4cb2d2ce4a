"""The C-ABI library loads and exports every declared entry point; host-side validation
rejects bad arguments before anything is launched (CPU only, no GPU calls)."""
from __future__ import annotations

import pytest

import paper_2606_21848_gb300 as kl
from paper_2606_21848_gb300 import _lib


@pytest.fixture(scope="module", autouse=True)
def built():
    kl.build()
    kl.load()


def test_every_declared_symbol_is_exported():
    names = _lib.declared_symbols()
    assert {"kl_route_query", "kl_append_v", "kl_decode_attention", "kl_combine",
            "kl_decode_workspace_size", "kl_status_string"} <= set(names)
    lib = kl.load()
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_header_constants_match_the_binding():
    """Every KL_* value the header defines (flags, statuses, dtypes, kernel choices) has the same
    value in the Python binding, so a flag added to one side cannot drift from the other."""
    import re
    text = open(_lib.HEADER).read()
    defined = {m.group(1): int(m.group(2), 0)
               for m in re.finditer(r"#define\s+(KL_FLAG_\w+)\s+(0x[0-9a-fA-F]+|\d+)", text)}
    for body in re.findall(r"typedef enum\s+\w*\s*\{(.*?)\}", text, re.S):
        for m in re.finditer(r"(KL_\w+)\s*=\s*(\d+)", body):
            defined[m.group(1)] = int(m.group(2))
    assert {"KL_FLAG_RANGE", "KL_FLAG_TIMEOUT", "KL_ERR_CUDA", "KL_FP32"} <= set(defined)
    wrong = {k: (v, getattr(_lib, k, None)) for k, v in defined.items() if getattr(_lib, k, None) != v}
    assert not wrong, wrong


def test_status_strings():
    assert kl.kl_status_string(kl.KL_OK) == "ok"
    assert "workspace" in kl.kl_status_string(kl.KL_ERR_WORKSPACE)
    assert kl.kl_status_string(99) == "unknown status"


def _shape(**kw):
    d = dict(num_seqs=2, num_q_heads=8, num_kv_heads=2, head_dim=128, page_size=16,
             num_pages=64, max_pages_per_seq=32)
    d.update(kw)
    return kl.make_shape(**d)


@pytest.mark.parametrize("kw,status", [
    (dict(num_kv_heads=3), kl.KL_ERR_INVALID_ARG),     # Hq not a multiple of Hkv
    (dict(head_dim=96), kl.KL_ERR_UNSUPPORTED),
    (dict(page_size=0), kl.KL_ERR_INVALID_ARG),
    (dict(num_pages=0), kl.KL_ERR_INVALID_ARG),
    (dict(num_seqs=-1), kl.KL_ERR_INVALID_ARG),
])
def test_bad_shapes_are_rejected_without_launch(kw, status):
    with pytest.raises(kl.KLError) as e:
        kl.kl_decode_attention(_shape(**kw), 16, 16, 16, 16, 16, 0, 16, kl.KL_FP32, None, stream=0)
    assert e.value.status == status
    with pytest.raises(kl.KLError):
        kl.kl_append_v(_shape(**kw), 16, 16, 16, 16, stream=0)


def test_null_pointers_are_rejected():
    with pytest.raises(kl.KLError) as e:
        kl.kl_decode_attention(_shape(), None, 16, 16, 16, 16, 1, 16, kl.KL_FP32, None, stream=0)
    assert e.value.status == kl.KL_ERR_INVALID_ARG
    with pytest.raises(kl.KLError):
        kl.kl_route_query(_shape(), 16, None, 16, stream=0)
    with pytest.raises(kl.KLError):
        kl.kl_combine(_shape(), None, 16, 4, 16, kl.KL_FP32, stream=0)


def test_workspace_too_small_is_rejected():
    sh = _shape(max_pages_per_seq=256)
    need = kl.kl_decode_workspace_size(sh, 8)
    assert need > 0
    assert kl.kl_decode_num_splits(sh, 8) == 8
    with pytest.raises(kl.KLError) as e:
        kl.kl_decode_attention(sh, 16, 16, 16, 16, 16, 8, 16, kl.KL_FP32, None, stream=0)
    assert e.value.status == kl.KL_ERR_WORKSPACE


def test_split_plan():
    sh = _shape(max_pages_per_seq=8192)                     # 131072 tokens
    assert kl.kl_decode_num_splits(sh, 128) == 128
    assert kl.kl_decode_workspace_size(sh, 128) >= 2 * 8 * 128 * (128 + 2) * 4
    assert kl.kl_decode_num_splits(sh, 1) == 1
    assert kl.kl_decode_workspace_size(sh, 1) == 0          # single split writes out directly
    small = _shape(max_pages_per_seq=16)                    # 256 tokens: quantum of 128 tokens
    assert kl.kl_decode_num_splits(small, 7) == 2
    assert kl.kl_decode_num_splits(sh, 0) >= 1
