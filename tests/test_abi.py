"""The C-ABI library loads and exports every symbol its headers declare; the
host-side argument checks work without a GPU."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for h in ("dllm.h", "dllm_ops.h"):
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names |= set(re.findall(r"\b(dllm_\w+)\s*\(", src))
    return names


@pytest.fixture(scope="module")
def libdllm():
    from paper_2606_13740_gb300 import build
    path = build()
    return C.CDLL(path)


def test_every_declared_symbol_is_exported(libdllm):
    names = _declared()
    assert {"dllm_init", "dllm_prefill", "dllm_denoise_step", "dllm_generate", "dllm_op_gemm"} <= names
    missing = [n for n in sorted(names) if not hasattr(libdllm, n)]
    assert not missing, missing


def test_binding_covers_every_symbol():
    from paper_2606_13740_gb300 import dllm
    assert _declared() == set(dllm.SIGNATURES)


def test_arena_bytes_and_config_checks():
    from paper_2606_13740_gb300 import Config, DllmError, dllm_arena_bytes
    tiny = dllm_arena_bytes(Config())
    assert tiny > 0
    big = dllm_arena_bytes(Config(n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464,
                                  mask_id=126463, rope_base=500000.0, max_ctx=1024, max_window=512))
    assert 15e9 < big < 40e9  # 15 GB of bf16 weights plus cache and scratch
    with pytest.raises(DllmError) as e:
        dllm_arena_bytes(Config(head_dim=96))
    assert "head_dim" in str(e.value)
    with pytest.raises(DllmError):
        dllm_arena_bytes(Config(mask_id=5000))
    with pytest.raises(DllmError):
        dllm_arena_bytes(Config(max_batch=64, max_window=128))


def test_init_without_gpu_reports_cuda_error():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    from paper_2606_13740_gb300 import dllm
    c = dllm.Config().c()
    h = C.c_void_p()
    rc = dllm.lib().dllm_init(C.byref(c), None, 0, None, C.byref(h))
    assert rc == -3 and not h.value
    assert b"CUDA" in dllm.lib().dllm_last_error(None) or len(dllm.lib().dllm_last_error(None)) > 0
