"""Python binding of the C ABI in ``include/dllm.h`` / ``include/dllm_ops.h``.

Argument marshalling only: every step of the denoising path runs in the CUDA
library's own kernels.  PyTorch serves as the device-memory and stream
provider (the arena is a torch CUDA tensor, the stream torch's current one).
The library must be built (``build()``); there is no fallback.
"""
from __future__ import annotations

import ctypes as C
import os
from dataclasses import dataclass

import numpy as np

from .build import OUT as _LIB_PATH
from .build import build as _build_lib

DLLM_OK, DLLM_DONE = 0, 1
ERRORS = {-1: "EINVAL", -2: "ENOMEM", -3: "ECUDA", -4: "ETIMEOUT", -5: "ESTATE", -6: "ECAPACITY"}
FIXED, MASKED, COMMITTED, STABLE, DRAFT = 0, 1, 2, 3, 4
COMMIT_SCHEDULE, COMMIT_THRESHOLD = 0, 1  # dllm_sched.commit_mode


class DllmError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"{ERRORS.get(code, code)}: {msg}")
        self.code = code


class dllm_config(C.Structure):
    _fields_ = [("n_layers", C.c_int), ("d_model", C.c_int), ("n_heads", C.c_int), ("head_dim", C.c_int),
                ("ffn", C.c_int), ("vocab", C.c_int), ("mask_id", C.c_int), ("rope_base", C.c_float),
                ("rms_eps", C.c_float), ("max_batch", C.c_int), ("max_ctx", C.c_int), ("max_window", C.c_int),
                ("block_len", C.c_int), ("weight_seed", C.c_uint64), ("n_kv_heads", C.c_int),
                ("weight_bits", C.c_int)]


class dllm_sched(C.Structure):
    _fields_ = [("steps_per_block", C.c_int), ("theta_remask", C.c_float), ("theta_stable", C.c_float),
                ("remask_max", C.c_int), ("spec_trigger", C.c_int), ("spec_blocks", C.c_int),
                ("use_prefix_cache", C.c_int), ("commit_mode", C.c_int), ("theta_visible", C.c_float),
                ("scr_rows", C.c_int), ("spec_allowance", C.c_float), ("spec_lat_n", C.c_int),
                ("spec_lat", C.c_float * 8), ("sls", C.c_int), ("slide", C.c_int)]


class dllm_step_out(C.Structure):
    _fields_ = [("n_committed", C.c_int), ("n_remasked", C.c_int), ("n_stable", C.c_int), ("n_drafts", C.c_int),
                ("block_done", C.c_int), ("masked_after", C.c_int), ("n_refreshed", C.c_int), ("n_revised", C.c_int)]

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_}


class dllm_stats(C.Structure):
    _fields_ = [("steps", C.c_int), ("spec_steps", C.c_int), ("blocks", C.c_int)]


# name -> (restype, argtypes); every entry point of include/dllm.h and dllm_ops.h
_P, _I, _F, _U64, _SZ = C.c_void_p, C.c_int, C.c_float, C.c_uint64, C.c_size_t
SIGNATURES = {
    "dllm_arena_bytes": (_I, [_P, C.POINTER(_SZ)]),
    "dllm_init": (_I, [_P, _P, _SZ, _P, C.POINTER(_P)]),
    "dllm_free": (None, [_P]),
    "dllm_last_error": (C.c_char_p, [_P]),
    "dllm_sync": (_I, [_P]),
    "dllm_prefill": (_I, [_P, _P, _I, _P, _I, _I]),
    "dllm_set_prefix_kv_random": (_I, [_P, _P, _I, _I, _I, _U64]),
    "dllm_begin_block": (_I, [_P]),
    "dllm_denoise_step": (_I, [_P, _P]),
    "dllm_rewind_block": (_I, [_P]),
    "dllm_generate": (_I, [_P, _P, _I, _P, _I, _I, _P, _P]),
    "dllm_window": (_I, [_P, _P]),
    "dllm_get_state": (_I, [_P, _P, _P, _P]),
    "dllm_set_state": (_I, [_P, _P, _P]),
    "dllm_get_step_debug": (_I, [_P, _P, _P, _P, _P]),
    "dllm_get_scr_debug": (_I, [_P, _P, _P, _P, _P, _P]),
    "dllm_set_debug": (_I, [_P, _I]),
    "dllm_get_weight": (_I, [_P, _I, _I, _P, _SZ]),
    "dllm_get_kv": (_I, [_P, _I, _I, _I, _I, _I, _P]),
    "dllm_set_profile": (_I, [_P, _I]),
    "dllm_get_profile": (_I, [_P, _P, _P, _P]),
    "dllm_launches_per_step": (_I, [_P, _P]),
    "dllm_get_trace": (_I, [_P, _P, _I, _P]),
    "dllm_op_gemm": (_I, [_P, _P, _P, _I, _I, _I, _I, _P]),
    "dllm_op_gemm_noalloc": (_I, [_P, _P, _P, _I, _I, _I, _I, _P]),
    "dllm_op_gemm_trace": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _P, _P, _P, _P]),
    "dllm_op_gemm_timed": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P]),
    "dllm_op_attention": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _P]),
    "dllm_op_lmhead": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _P]),
    "dllm_op_commit": (_I, [_P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P, _I, _F, _F, _I, _I, _I, _I, _I, _I, _F, _P]),
}

_lib = None


def lib(build_if_missing: bool = True):
    """Load libdllm.so (building it first if asked); raises if unavailable."""
    global _lib
    if _lib is None:
        path = _LIB_PATH
        if build_if_missing:
            path = _build_lib()
        if not os.path.exists(path):
            raise RuntimeError(f"CUDA library not built: {path}")
        L = C.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _p(a):
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        return a.ctypes.data_as(C.c_void_p)
    return C.c_void_p(int(a))


def _check(rc, ctx=None):
    if rc < 0:
        msg = lib().dllm_last_error(ctx).decode(errors="replace")
        raise DllmError(rc, msg)
    return rc


@dataclass
class Config:
    n_layers: int = 2
    d_model: int = 256
    n_heads: int = 4
    head_dim: int = 64
    ffn: int = 688
    vocab: int = 1024
    mask_id: int = 1023
    rope_base: float = 10000.0
    rms_eps: float = 1e-5
    max_batch: int = 1
    max_ctx: int = 256
    max_window: int = 128
    block_len: int = 32
    weight_seed: int = 0x11ADA8B
    n_kv_heads: int = 0  # grouped-query attention: K/V heads (0 = n_heads)
    weight_bits: int = 16  # 4: projections in the 4-bit block format (Q4_0 weights, Sec. 5.1)

    @property
    def kv_dim(self):
        return (self.n_kv_heads or self.n_heads) * self.head_dim

    def c(self):
        return dllm_config(self.n_layers, self.d_model, self.n_heads, self.head_dim, self.ffn, self.vocab,
                           self.mask_id, self.rope_base, self.rms_eps, self.max_batch, self.max_ctx, self.max_window,
                           self.block_len, self.weight_seed, self.n_kv_heads, self.weight_bits)


@dataclass
class Sched:
    steps_per_block: int = 8
    theta_remask: float = 0.0
    theta_stable: float = 0.9
    remask_max: int = 1
    spec_trigger: int = 8
    spec_blocks: int = 0
    use_prefix_cache: int = 1
    commit_mode: int = COMMIT_SCHEDULE
    theta_visible: float = 0.7
    scr_rows: int = 0  # sparse cache refresh: visible prefix positions re-scored per step (one sequence)
    spec_allowance: float = -1.0  # adaptive lookahead allowance (< 0: fixed, all spec_blocks)
    spec_lat: tuple = ()          # step latency with a window of 1, 2, ... blocks (at most 8)
    sls: int = 0                  # selective logits skipping: the LM head only for rows needing a decision
    slide: int = 0                # continuous sliding of the window along the commit frontier (batch 1)

    def c(self):
        lat = (C.c_float * 8)(*self.spec_lat[:8])
        return dllm_sched(self.steps_per_block, self.theta_remask, self.theta_stable, self.remask_max,
                          self.spec_trigger, self.spec_blocks, self.use_prefix_cache, self.commit_mode,
                          self.theta_visible, self.scr_rows, self.spec_allowance, len(self.spec_lat[:8]), lat,
                          self.sls, self.slide)


def dllm_arena_bytes(cfg: Config) -> int:
    n = C.c_size_t()
    c = cfg.c()
    _check(lib().dllm_arena_bytes(C.byref(c), C.byref(n)))
    return n.value


class Context:
    """A dllm_ctx on the current CUDA device; the arena is a torch tensor."""

    def __init__(self, cfg: Config, use_torch_arena: bool = True, stream=None):
        import torch

        self.cfg = cfg
        self._c = cfg.c()
        nbytes = dllm_arena_bytes(cfg)
        self.arena = None
        arena_ptr = None
        if use_torch_arena:
            self.arena = torch.empty(nbytes + 256, dtype=torch.uint8, device="cuda")
            arena_ptr = (self.arena.data_ptr() + 255) // 256 * 256
        if stream is None:
            # a stream of its own: torch's default stream is the legacy stream
            # (handle 0), which the C ABI would read as "create one"
            stream = torch.cuda.Stream()
        self.stream = stream
        h = C.c_void_p()
        _check(lib().dllm_init(C.byref(self._c), _p(arena_ptr), nbytes, _p(stream.cuda_stream), C.byref(h)))
        self.h = h
        self.B = 0
        self.n_pos = 0
        self.Lp = 0

    # -- thin wrappers with the ABI's names -------------------------------------------------------
    def dllm_prefill(self, sched: Sched, prompt, gen_len):
        prompt = np.ascontiguousarray(np.atleast_2d(prompt), np.int32)
        self._s = sched.c()
        B, Lp = prompt.shape
        _check(lib().dllm_prefill(self.h, C.byref(self._s), B, _p(prompt), Lp, gen_len), self.h)
        self.B, self.Lp, self.n_pos = B, Lp, Lp + gen_len

    def dllm_set_prefix_kv_random(self, sched: Sched, batch, P, gen_len, seed):
        self._s = sched.c()
        _check(lib().dllm_set_prefix_kv_random(self.h, C.byref(self._s), batch, P, gen_len, seed), self.h)
        self.B, self.Lp, self.n_pos = batch, P, P + gen_len

    def dllm_begin_block(self) -> bool:
        rc = _check(lib().dllm_begin_block(self.h), self.h)
        return rc == DLLM_OK

    def dllm_denoise_step(self, want_out=True):
        out = dllm_step_out()
        _check(lib().dllm_denoise_step(self.h, C.byref(out) if want_out else None), self.h)
        return out.as_dict() if want_out else None

    def dllm_rewind_block(self):
        _check(lib().dllm_rewind_block(self.h), self.h)

    def dllm_generate(self, sched: Sched, prompt, gen_len):
        prompt = np.ascontiguousarray(np.atleast_2d(prompt), np.int32)
        B, Lp = prompt.shape
        out = np.empty((B, gen_len), np.int32)
        st = dllm_stats()
        self._s = sched.c()
        _check(lib().dllm_generate(self.h, C.byref(self._s), B, _p(prompt), Lp, gen_len, _p(out), C.byref(st)),
               self.h)
        self.B, self.Lp, self.n_pos = B, Lp, Lp + gen_len
        return out, {k: getattr(st, k) for k, _ in st._fields_}

    def dllm_window(self):
        info = np.zeros(7, np.int32)
        _check(lib().dllm_window(self.h, _p(info)), self.h)
        return dict(zip(("w0", "T", "c0", "c1", "step", "kv_len", "spec_on"), (int(v) for v in info)))

    def dllm_get_state(self):
        tok = np.empty((self.B, self.n_pos), np.int32)
        st = np.empty((self.B, self.n_pos), np.uint8)
        kv = np.empty(self.B, np.int32)
        _check(lib().dllm_get_state(self.h, _p(tok), _p(st), _p(kv)), self.h)
        return tok, st, kv

    def dllm_set_state(self, tok=None, st=None):
        t = None if tok is None else np.ascontiguousarray(np.reshape(tok, (self.B, self.n_pos)), np.int32)
        s = None if st is None else np.ascontiguousarray(np.reshape(st, (self.B, self.n_pos)), np.uint8)
        _check(lib().dllm_set_state(self.h, _p(t), _p(s)), self.h)

    def dllm_set_debug(self, flags):
        _check(lib().dllm_set_debug(self.h, flags), self.h)

    def dllm_get_step_debug(self, logits=False):
        T = self.dllm_window()["T"]
        n = self.B * T
        x0 = np.empty(n, np.int32)
        conf = np.empty(n, np.float32)
        tc = np.empty(n, np.float32)
        lg = np.empty((n, self.cfg.vocab), np.float32) if logits else None
        _check(lib().dllm_get_step_debug(self.h, _p(lg), _p(x0), _p(conf), _p(tc)), self.h)
        r = {"x0": x0.reshape(self.B, T), "conf": conf.reshape(self.B, T), "tokconf": tc.reshape(self.B, T)}
        if logits:
            r["logits"] = lg.reshape(self.B, T, self.cfg.vocab)
        return r

    def dllm_get_scr_debug(self, seq=0):
        """The last step's sparse-cache-refresh rows of sequence seq: positions (-1 unused),
        argmax, conf, tokconf."""
        n = C.c_int()
        _check(lib().dllm_get_scr_debug(self.h, None, None, None, None, C.byref(n)), self.h)
        k = max(1, n.value)
        pos = np.empty((self.B, k), np.int32)
        x0 = np.empty((self.B, k), np.int32)
        conf = np.empty((self.B, k), np.float32)
        tc = np.empty((self.B, k), np.float32)
        _check(lib().dllm_get_scr_debug(self.h, _p(pos), _p(x0), _p(conf), _p(tc), C.byref(n)), self.h)
        k = n.value
        return {"pos": pos[seq, :k], "x0": x0[seq, :k], "conf": conf[seq, :k], "tokconf": tc[seq, :k]}

    def dllm_get_weight(self, layer, which):
        c = self.cfg
        qd = c.n_heads * c.head_dim
        shapes = {0: (qd, c.d_model), 1: (c.kv_dim, c.d_model), 2: (c.kv_dim, c.d_model), 3: (c.d_model, qd),
                  4: (c.ffn, c.d_model), 5: (c.ffn, c.d_model), 6: (c.d_model, c.ffn)}
        shape = (c.vocab, c.d_model) if layer < 0 else shapes[which]
        out = np.empty(shape, np.uint16)
        _check(lib().dllm_get_weight(self.h, layer, which, _p(out), out.size), self.h)
        return out

    def dllm_get_kv(self, layer, which, seq, p0, n):
        out = np.empty((n, self.cfg.kv_dim), np.float32)
        _check(lib().dllm_get_kv(self.h, layer, which, seq, p0, n, _p(out)), self.h)
        return out

    KINDS = ("embed", "norm", "qkv", "attn", "oproj", "gateup", "down", "head", "head_reduce", "commit", "layer")

    def dllm_set_profile(self, enable):
        _check(lib().dllm_set_profile(self.h, int(enable)), self.h)

    def dllm_get_profile(self):
        ms = np.zeros(len(self.KINDS), np.float64)
        launches = np.zeros(len(self.KINDS), np.int32)
        steps = np.zeros(1, np.int32)
        _check(lib().dllm_get_profile(self.h, _p(ms), _p(launches), _p(steps)), self.h)
        return {k: {"ms_total": float(ms[i]), "launches_per_step": int(launches[i])} for i, k in
                enumerate(self.KINDS)}, int(steps[0])

    def dllm_get_trace(self, max_launches=512):
        out = np.zeros((max_launches, 256, 16), np.uint64)
        n = np.zeros(1, np.int32)
        _check(lib().dllm_get_trace(self.h, _p(out), max_launches, _p(n)), self.h)
        return out[: int(n[0])]

    def dllm_launches_per_step(self):
        n = np.zeros(1, np.int32)
        _check(lib().dllm_launches_per_step(self.h, _p(n)), self.h)
        return int(n[0])

    def dllm_sync(self):
        _check(lib().dllm_sync(self.h), self.h)

    def close(self):
        if getattr(self, "h", None):
            lib().dllm_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# -- single-kernel entry points ------------------------------------------------------------------
def _stream_ptr(stream):
    return None if stream is None else stream.cuda_stream


def dllm_op_gemm(W, X, M, N, K, grid=0, stream=None):
    """W, X torch bf16 CUDA tensors; returns D fp32 [N][M]."""
    import torch

    D = torch.empty((N, M), dtype=torch.float32, device=W.device)
    _check(lib().dllm_op_gemm(_p(W.data_ptr()), _p(X.data_ptr()), _p(D.data_ptr()), M, N, K, grid,
                              _p(_stream_ptr(stream))))
    return D


def dllm_op_gemm_noalloc(W, X, D, M, N, K, grid=0, stream=None):
    """dllm_op_gemm into a caller-provided D (fp32 [N][M]); allocates nothing."""
    _check(lib().dllm_op_gemm_noalloc(_p(W.data_ptr()), _p(X.data_ptr()), _p(D.data_ptr()), M, N, K, grid,
                                      _p(_stream_ptr(stream))))
    return D


def dllm_op_gemm_timed(W, X, M, N, K, reps, grid=0, flags=0, stream=None):
    """Average kernel time (ms) of `reps` back-to-back launches, and D (flags: see dllm_ops.h)."""
    import torch

    D = torch.empty((N, M), dtype=torch.float32, device=W.device)
    ms = C.c_float()
    _check(lib().dllm_op_gemm_timed(_p(W.data_ptr()), _p(X.data_ptr()), _p(D.data_ptr()), M, N, K, grid, reps,
                                    flags, C.byref(ms), _p(_stream_ptr(stream))))
    return ms.value, D


def dllm_op_gemm_trace(W, X, M, N, K, reps, grid=0, stream=None):
    """(ms per launch, per-CTA timeline [grid][8] of the last launch)."""
    import torch

    D = torch.empty((N, M), dtype=torch.float32, device=W.device)
    ms = C.c_float()
    used = C.c_int()
    tr = np.zeros((1024, 16), np.uint64)
    _check(lib().dllm_op_gemm_trace(_p(W.data_ptr()), _p(X.data_ptr()), _p(D.data_ptr()), M, N, K, grid, reps,
                                    C.byref(ms), _p(tr), C.byref(used), _p(_stream_ptr(stream))))
    return ms.value, tr[:used.value]


def dllm_op_attention(q, kc, vc, kv_len, B, T, H, hd, cap, max_kv_len, stream=None, Hkv=None):
    """q bf16 [B][H][T][hd], kc/vc bf16 [B][Hkv][cap][hd] (Hkv defaults to H); returns bf16 [B*T][H*hd]."""
    import torch

    out = torch.empty((B * T, H * hd), dtype=torch.bfloat16, device=q.device)
    _check(lib().dllm_op_attention(_p(q.data_ptr()), _p(kc.data_ptr()), _p(vc.data_ptr()), _p(kv_len.data_ptr()),
                                   _p(out.data_ptr()), B, T, H, H if Hkv is None else Hkv, hd, cap, max_kv_len,
                                   _p(_stream_ptr(stream))))
    return out


def dllm_op_lmhead(W, X, cur, V, N, d, mask_id, want_logits=False, stream=None):
    import torch

    dev = W.device
    x0 = torch.empty(N, dtype=torch.int32, device=dev)
    conf = torch.empty(N, dtype=torch.float32, device=dev)
    tc = torch.empty(N, dtype=torch.float32, device=dev)
    lg = torch.empty((N, V), dtype=torch.float32, device=dev) if want_logits else None
    _check(lib().dllm_op_lmhead(_p(W.data_ptr()), _p(X.data_ptr()), _p(cur.data_ptr()), _p(x0.data_ptr()),
                                _p(conf.data_ptr()), _p(tc.data_ptr()), _p(None if lg is None else lg.data_ptr()),
                                V, N, d, mask_id, _p(_stream_ptr(stream))))
    return x0, conf, tc, lg


def dllm_op_commit(sched: Sched, mask_id, tok, st, w0, T, c0, c1, step, x0, conf, tokconf, block_len=32):
    tok = np.ascontiguousarray(tok, np.int32).copy()
    st = np.ascontiguousarray(st, np.uint8).copy()
    x0 = np.ascontiguousarray(x0, np.int32)
    conf = np.ascontiguousarray(conf, np.float32)
    tokconf = np.ascontiguousarray(tokconf, np.float32)
    out = np.zeros(6, np.int32)
    _check(lib().dllm_op_commit(_p(tok), _p(st), tok.size, w0, T, c0, c1, step, _p(x0), _p(conf), _p(tokconf),
                                sched.steps_per_block, sched.theta_remask, sched.theta_stable, sched.remask_max,
                                sched.spec_blocks, sched.use_prefix_cache, block_len, mask_id, sched.commit_mode,
                                sched.theta_visible, _p(out)))
    keys = ("n_committed", "n_remasked", "n_stable", "n_drafts", "block_done", "masked_after")
    return tok, st, dict(zip(keys, (int(v) for v in out)))
