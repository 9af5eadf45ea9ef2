"""CPU oracle for block-wise diffusion-LLM decoding (arXiv 2606.13740).

Test infrastructure only: the test suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg use it; the product path never does.  It shares
no code with the CUDA library.
"""
from .oracle import (  # noqa: F401
    MASKED, COMMITTED, STABLE, DRAFT, FIXED,
    OracleConfig, OracleSched, Model, Session, build, lib, commit, decide,
    gen_bf16, gen_f32, bf16_to_f32, f32_to_bf16_bits, rmsnorm, rope, forward,
    q4_dequant, q4_code, q4_scale, gen_q4,
    W_Q, W_K, W_V, W_O, W_GATE, W_UP, W_DOWN, T_EMBED, T_HEAD,
)
