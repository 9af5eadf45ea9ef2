"""GB300 (sm_103a) block-wise diffusion-LLM denoising path.

Implements the repeated denoising step of "Efficient On-Device Diffusion LLM
Inference with Mobile NPU" (arXiv 2606.13740): a bidirectional LLaDA forward
over the current block (plus draft tokens of future blocks) against a frozen
prefix KV cache, followed by confidence-based commit, re-mask and drafting.
The compute lives in ``libdllm.so`` (hand-written CUDA); this package is its
ctypes binding.
"""
from .build import build  # noqa: F401
from .dllm import (  # noqa: F401
    COMMIT_SCHEDULE, COMMIT_THRESHOLD, COMMITTED, DRAFT, FIXED, MASKED, STABLE, Config, Context, DllmError, Sched,
    dllm_arena_bytes, dllm_op_attention,
    dllm_op_commit, dllm_op_gemm, dllm_op_lmhead, lib,
)
