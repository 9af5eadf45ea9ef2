"""ctypes wrapper of the C oracle (``dllm_oracle.c``).

Test infrastructure only (see the package docstring).  ``build()`` compiles
the C source with gcc into ``liboracle.so`` next to it; the flags keep every
floating-point operation of the weight generator a single IEEE rounding
(``-ffp-contract=off``).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from dataclasses import dataclass

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "dllm_oracle.c")
LIB = os.path.join(HERE, "liboracle.so")

FIXED, MASKED, COMMITTED, STABLE, DRAFT = 0, 1, 2, 3, 4
W_Q, W_K, W_V, W_O, W_GATE, W_UP, W_DOWN = range(7)
T_EMBED, T_HEAD = 1, 2


def build(force: bool = False) -> str:
    """Compile the oracle shared library (gcc + OpenMP)."""
    hdr = os.path.join(HERE, "dllm_oracle.h")
    if (not force and os.path.exists(LIB)
            and os.path.getmtime(LIB) >= max(os.path.getmtime(SRC), os.path.getmtime(hdr))):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared", "-std=c11",
           "-o", tmp, SRC, "-lm"]
    subprocess.check_call(cmd)
    os.replace(tmp, LIB)
    return LIB


class _Cfg(C.Structure):
    _fields_ = [("n_layers", C.c_int), ("d_model", C.c_int), ("n_heads", C.c_int),
                ("head_dim", C.c_int), ("ffn", C.c_int), ("vocab", C.c_int), ("mask_id", C.c_int),
                ("rope_base", C.c_double), ("rms_eps", C.c_double), ("weight_seed", C.c_uint64),
                ("n_kv_heads", C.c_int), ("weight_bits", C.c_int)]


class _Sched(C.Structure):
    _fields_ = [("steps_per_block", C.c_int), ("block_len", C.c_int), ("theta_remask", C.c_float),
                ("theta_stable", C.c_float), ("remask_max", C.c_int), ("spec_trigger", C.c_int),
                ("spec_blocks", C.c_int), ("use_prefix_cache", C.c_int), ("commit_mode", C.c_int),
                ("theta_visible", C.c_float), ("scr_rows", C.c_int), ("spec_allowance", C.c_float),
                ("spec_lat_n", C.c_int), ("spec_lat", C.c_float * 8), ("slide", C.c_int)]


class _StepOut(C.Structure):
    _fields_ = [("n_committed", C.c_int), ("n_remasked", C.c_int), ("n_stable", C.c_int),
                ("n_drafts", C.c_int), ("block_done", C.c_int), ("masked_after", C.c_int),
                ("n_refreshed", C.c_int), ("n_revised", C.c_int)]

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_}


_lib = None


def lib():
    global _lib
    if _lib is None:
        build()
        L = C.CDLL(LIB)
        P, I, U64, D, F = C.c_void_p, C.c_int, C.c_uint64, C.c_double, C.c_float
        L.orc_splitmix_at.restype = U64
        L.orc_splitmix_at.argtypes = [U64, U64]
        L.orc_gen_f32.argtypes = [U64, U64, U64, U64, D, P]
        L.orc_gen_bf16.argtypes = [U64, U64, U64, U64, D, P]
        L.orc_f32_to_bf16.restype = C.c_uint16
        L.orc_f32_to_bf16.argtypes = [F]
        L.orc_q4_dequant.restype = C.c_uint16
        L.orc_q4_dequant.argtypes = [I, C.c_uint16]
        L.orc_q4_code.restype = I
        L.orc_q4_code.argtypes = [U64, U64, I, I, I]
        L.orc_q4_scale.restype = C.c_uint16
        L.orc_q4_scale.argtypes = [U64, U64, I, I, I]
        L.orc_gen_q4.argtypes = [U64, U64, I, I, P]
        L.orc_model_new.restype = P
        L.orc_model_new.argtypes = [P, I, I]
        L.orc_model_new_zero.restype = P
        L.orc_model_new_zero.argtypes = [P]
        L.orc_model_weight.restype = P
        L.orc_model_weight.argtypes = [P, I, I, C.POINTER(C.c_size_t)]
        L.orc_model_norm.restype = P
        L.orc_model_norm.argtypes = [P, I, I]
        L.orc_model_free.argtypes = [P]
        L.orc_rmsnorm.argtypes = [I, P, P, D, P]
        L.orc_rope.argtypes = [I, D, I, P]
        L.orc_decide.argtypes = [I, I, P, C.c_int32, P, P, P, P]
        L.orc_forward.restype = I
        L.orc_forward.argtypes = [P, I, P, P, I, P, P, P, P, P, P, I]
        L.orc_commit.restype = I
        L.orc_commit.argtypes = [P, I, I, P, P, I, I, I, I, I, P, P, P, P]
        L.orc_session_new.restype = P
        L.orc_session_new.argtypes = [P, P, I, P, I]
        L.orc_session_free.argtypes = [P]
        for fn in ("orc_prefill", "orc_begin_block"):
            getattr(L, fn).restype = I
            getattr(L, fn).argtypes = [P]
        L.orc_denoise_step.restype = I
        L.orc_denoise_step.argtypes = [P, P, I]
        L.orc_window.argtypes = [P, P]
        L.orc_step_decisions.restype = I
        L.orc_step_decisions.argtypes = [P, P, P, P, P, P]
        L.orc_scr_decisions.restype = I
        L.orc_scr_decisions.argtypes = [P, P, P, P, P, P]
        L.orc_get_state.argtypes = [P, P, P, P]
        L.orc_set_state.argtypes = [P, P, P]
        L.orc_prefix_kv.restype = P
        L.orc_prefix_kv.argtypes = [P, I, I]
        L.orc_n_pos.restype = I
        L.orc_n_pos.argtypes = [P]
        _lib = L
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


@dataclass
class OracleConfig:
    n_layers: int = 2
    d_model: int = 256
    n_heads: int = 4
    head_dim: int = 64
    ffn: int = 688
    vocab: int = 1024
    mask_id: int = 1023
    rope_base: float = 10000.0
    rms_eps: float = 1e-5
    weight_seed: int = 0x11ADA8B
    n_kv_heads: int = 0  # grouped-query attention (Dream-7B style); 0 = n_heads (LLaDA's multi-head)
    weight_bits: int = 16  # 4: the projections in the 4-bit block format (Q4_0, Sec. 5.1)

    @property
    def kv_dim(self):
        return (self.n_kv_heads or self.n_heads) * self.head_dim

    def c(self):
        return _Cfg(self.n_layers, self.d_model, self.n_heads, self.head_dim, self.ffn, self.vocab,
                    self.mask_id, self.rope_base, self.rms_eps, self.weight_seed, self.n_kv_heads,
                    self.weight_bits)


@dataclass
class OracleSched:
    steps_per_block: int = 8
    block_len: int = 32
    theta_remask: float = 0.0
    theta_stable: float = 0.9
    remask_max: int = 1
    spec_trigger: int = 8
    spec_blocks: int = 0
    use_prefix_cache: int = 1
    commit_mode: int = 0          # 0: LLaDA's fixed schedule; 1: threshold (staged stabilization)
    theta_visible: float = 0.7
    scr_rows: int = 0             # sparse cache refresh: visible prefix positions re-scored per step
    spec_allowance: float = -1.0  # adaptive lookahead allowance (< 0: fixed, all spec_blocks)
    spec_lat: tuple = ()          # step latency with a window of 1, 2, ... blocks (at most 8)
    slide: int = 0                # continuous sliding of the window along the commit frontier

    def c(self):
        lat = (C.c_float * 8)(*self.spec_lat[:8])
        return _Sched(self.steps_per_block, self.block_len, self.theta_remask, self.theta_stable,
                      self.remask_max, self.spec_trigger, self.spec_blocks, self.use_prefix_cache,
                      self.commit_mode, self.theta_visible, self.scr_rows, self.spec_allowance,
                      len(self.spec_lat[:8]), lat, self.slide)


def gen_f32(seed, tensor_id, first, n, sigma):
    out = np.empty(n, np.float32)
    lib().orc_gen_f32(seed, tensor_id, first, n, sigma, _p(out))
    return out


def gen_bf16(seed, tensor_id, first, n, sigma):
    out = np.empty(n, np.uint16)
    lib().orc_gen_bf16(seed, tensor_id, first, n, sigma, _p(out))
    return out


def q4_dequant(code, scale_bits):
    """bf16 bits of the 4-bit block format's weight d * (code - 8) (orc_q4_dequant)."""
    return int(lib().orc_q4_dequant(int(code), int(scale_bits)))


def q4_code(seed, tid, cols, r, c):
    return int(lib().orc_q4_code(seed, tid, cols, r, c))


def q4_scale(seed, tid, cols, r, b):
    return int(lib().orc_q4_scale(seed, tid, cols, r, b))


def gen_q4(seed, tid, rows, cols):
    """rows x cols weights of tensor tid in the 4-bit format, as dequantised bf16 bits."""
    out = np.empty((rows, cols), np.uint16)
    lib().orc_gen_q4(seed, tid, rows, cols, _p(out))
    return out


def bf16_to_f32(bits):
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def f32_to_bf16_bits(x):
    L = lib()
    return np.array([L.orc_f32_to_bf16(float(v)) for v in np.asarray(x, np.float32).ravel()], np.uint16)


def rmsnorm(x, gamma, eps):
    x = np.ascontiguousarray(x, np.float32)
    gamma = np.ascontiguousarray(gamma, np.float32)
    out = np.empty_like(x)
    lib().orc_rmsnorm(x.size, _p(x), _p(gamma), eps, _p(out))
    return out


def rope(vec, base, pos):
    v = np.ascontiguousarray(vec, np.float32).copy()
    lib().orc_rope(v.size, base, pos, _p(v))
    return v


def decide(logits, mask_id, cur):
    z = np.ascontiguousarray(logits, np.float32)
    x0 = C.c_int32()
    conf, tokconf, margin = C.c_float(), C.c_float(), C.c_float()
    lib().orc_decide(z.size, mask_id, _p(z), int(cur), C.byref(x0), C.byref(conf), C.byref(tokconf),
                     C.byref(margin))
    return x0.value, conf.value, tokconf.value, margin.value


def commit(sched: OracleSched, mask_id, tok, st, w0, T, c0, c1, step, x0, conf, tokconf):
    """Run one commit pass on copies of (tok, st); returns (tok, st, out)."""
    tok = np.ascontiguousarray(tok, np.int32).copy()
    st = np.ascontiguousarray(st, np.uint8).copy()
    x0 = np.ascontiguousarray(x0, np.int32)
    conf = np.ascontiguousarray(conf, np.float32)
    tokconf = np.ascontiguousarray(tokconf, np.float32)
    out = _StepOut()
    s = sched.c()
    rc = lib().orc_commit(C.byref(s), mask_id, tok.size, _p(tok), _p(st), w0, T, c0, c1, step, _p(x0),
                          _p(conf), _p(tokconf), C.byref(out))
    if rc:
        raise RuntimeError(f"orc_commit failed: {rc}")
    return tok, st, out.as_dict()


class Model:
    """Oracle model; weights are generated from the seed or filled by tests."""

    def __init__(self, cfg: OracleConfig, gen_layers: int = -1, gen_head: bool = True, zero: bool = False):
        self.cfg = cfg
        self._c = cfg.c()
        L = lib()
        self.h = L.orc_model_new_zero(C.byref(self._c)) if zero else \
            L.orc_model_new(C.byref(self._c), gen_layers, int(gen_head))

    def weight(self, layer, which):
        """numpy view (bf16 bits, logical [rows][cols]) of a weight."""
        c = self.cfg
        n = C.c_size_t()
        ptr = lib().orc_model_weight(self.h, layer, which, C.byref(n))
        if not ptr:
            raise KeyError((layer, which))
        qd = c.n_heads * c.head_dim
        kvd = c.kv_dim
        shapes = {W_Q: (qd, c.d_model), W_K: (kvd, c.d_model), W_V: (kvd, c.d_model), W_O: (c.d_model, qd),
                  W_GATE: (c.ffn, c.d_model), W_UP: (c.ffn, c.d_model), W_DOWN: (c.d_model, c.ffn)}
        shape = (c.vocab, c.d_model) if layer < 0 else shapes[which]
        buf = (C.c_uint16 * n.value).from_address(ptr)
        return np.frombuffer(buf, np.uint16).reshape(shape)

    def norm(self, layer, which=0):
        ptr = lib().orc_model_norm(self.h, layer, which)
        buf = (C.c_float * self.cfg.d_model).from_address(ptr)
        return np.frombuffer(buf, np.float32)

    def __del__(self):
        if getattr(self, "h", None):
            lib().orc_model_free(self.h)
            self.h = None


def forward(model: Model, tok, pos, prefix_k=None, prefix_v=None, group=None, want_kv=False, logits=True,
            n_layers_run=-1):
    """orc_forward; returns dict(logits [T][V], k [L][T][kvd], v [L][T][kvd]) (kvd: K/V heads x head_dim)."""
    c = model.cfg
    tok = np.ascontiguousarray(tok, np.int32)
    pos = np.ascontiguousarray(pos, np.int32)
    T = tok.size
    kvd = c.kv_dim
    P = 0 if prefix_k is None else prefix_k.shape[1]
    pk = None if prefix_k is None else np.ascontiguousarray(prefix_k, np.float32)
    pv = None if prefix_v is None else np.ascontiguousarray(prefix_v, np.float32)
    grp = None if group is None else np.ascontiguousarray(group, np.int32)
    L = c.n_layers if n_layers_run < 0 else n_layers_run
    ok = np.empty((L, T, kvd), np.float32) if want_kv else None
    ov = np.empty((L, T, kvd), np.float32) if want_kv else None
    lg = np.empty((T, c.vocab), np.float32) if logits else None
    rc = lib().orc_forward(model.h, T, _p(tok), _p(pos), P, _p(pk), _p(pv), _p(grp), _p(ok), _p(ov), _p(lg),
                           n_layers_run)
    if rc:
        raise RuntimeError(f"orc_forward failed: {rc}")
    return {"logits": lg, "k": ok, "v": ov}


class Session:
    """One sequence's block-wise decoding state (prefill, blocks, steps)."""

    def __init__(self, model: Model, sched: OracleSched, prompt, gen_len):
        self.model = model
        self.sched = sched
        self._s = sched.c()
        prompt = np.ascontiguousarray(prompt, np.int32)
        self.Lp = prompt.size
        self.gen_len = gen_len
        self.h = lib().orc_session_new(model.h, C.byref(self._s), self.Lp, _p(prompt), gen_len)
        self.n_pos = lib().orc_n_pos(self.h)

    def prefill(self):
        rc = lib().orc_prefill(self.h)
        if rc:
            raise RuntimeError(rc)

    def begin_block(self) -> bool:
        rc = lib().orc_begin_block(self.h)
        if rc < 0:
            raise RuntimeError(f"orc_begin_block: {rc}")
        return rc == 0

    def step(self, keep_logits=False):
        out = _StepOut()
        rc = lib().orc_denoise_step(self.h, C.byref(out), int(keep_logits))
        if rc:
            raise RuntimeError(f"orc_denoise_step: {rc}")
        return out.as_dict()

    def window(self):
        info = np.zeros(7, np.int32)
        lib().orc_window(self.h, _p(info))
        keys = ("w0", "T", "c0", "c1", "step", "kv_len", "spec_on")
        return dict(zip(keys, (int(v) for v in info)))

    def decisions(self, logits=False):
        T = self.window()["T"]
        x0 = np.empty(T, np.int32)
        conf = np.empty(T, np.float32)
        tokconf = np.empty(T, np.float32)
        margin = np.empty(T, np.float32)
        lg = np.empty((T, self.model.cfg.vocab), np.float32) if logits else None
        rc = lib().orc_step_decisions(self.h, _p(x0), _p(conf), _p(tokconf), _p(margin), _p(lg))
        if rc:
            raise RuntimeError(rc)
        return {"x0": x0, "conf": conf, "tokconf": tokconf, "margin": margin, "logits": lg}

    def scr_decisions(self):
        """The last step's tracked prefix positions (sparse cache refresh) and their decisions."""
        R = max(1, self.sched.scr_rows)
        pos = np.empty(R, np.int32)
        x0 = np.empty(R, np.int32)
        conf = np.empty(R, np.float32)
        tokconf = np.empty(R, np.float32)
        margin = np.empty(R, np.float32)
        n = lib().orc_scr_decisions(self.h, _p(pos), _p(x0), _p(conf), _p(tokconf), _p(margin))
        return {"pos": pos[:n], "x0": x0[:n], "conf": conf[:n], "tokconf": tokconf[:n], "margin": margin[:n]}

    def state(self):
        tok = np.empty(self.n_pos, np.int32)
        st = np.empty(self.n_pos, np.uint8)
        kv = C.c_int32()
        lib().orc_get_state(self.h, _p(tok), _p(st), C.byref(kv))
        return tok, st, kv.value

    def set_state(self, tok, st):
        tok = np.ascontiguousarray(tok, np.int32)
        st = np.ascontiguousarray(st, np.uint8)
        lib().orc_set_state(self.h, _p(tok), _p(st))

    def prefix_kv(self, layer, which):
        c = self.model.cfg
        kv_len = self.state()[2]
        kvd = c.kv_dim
        ptr = lib().orc_prefix_kv(self.h, layer, which)
        buf = (C.c_float * (kv_len * kvd)).from_address(ptr)
        return np.frombuffer(buf, np.float32).reshape(kv_len, kvd).copy()

    def generate(self):
        """Whole block loop; returns the generated ids."""
        self.prefill()
        while self.begin_block():
            while True:
                o = self.step()
                if o["block_done"]:
                    break
        tok, _, _ = self.state()
        return tok[self.Lp:]

    def __del__(self):
        if getattr(self, "h", None):
            lib().orc_session_free(self.h)
            self.h = None
