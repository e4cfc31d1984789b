"""Urgency-Aware Denoising on GB300: Python binding of the C ABI in include/uad.h.

Argument marshalling only: every step of the denoising loop runs in the library's CUDA
kernels. There is no CPU fallback; importing this package fails if libuad.so is missing.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libuad.so")
if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with `python paper_2609_37772_gb300/build.py` "
                      "(or __graft_entry__.build()); there is no fallback path")
_lib = C.CDLL(LIB_PATH)

UAD_OK, UAD_EINVAL, UAD_ESTATE, UAD_ENOMEM, UAD_ECUDA, UAD_ETIMEDOUT, UAD_ENONFINITE = 0, -22, -1, -12, -5, -110, -33
KIND = {"adarms": 0, "dit": 1, "concat": 2}
DTYPE = {"f32": 0, "bf16": 1}
MAX_STEPS = 64

_I32, _P = C.c_int32, C.c_void_p


class uad_arch(C.Structure):
    _fields_ = [(n, _I32) for n in ("kind", "dtype", "n_layers", "width", "n_heads", "n_kv_heads",
                                    "head_dim", "mlp_dim", "action_dim", "chunk_len", "prefix_len",
                                    "prefix_width", "rope", "max_batch")]


class uad_schedule(C.Structure):
    _fields_ = [("budgets", C.POINTER(_I32)), ("batch", _I32), ("n_exec", _I32), ("tr", _I32),
                ("gac", _I32), ("chunk_relative", _I32), ("gac_mask", C.POINTER(C.c_uint8)),
                ("rot_dim", _I32)]


class uad_stats(C.Structure):
    _fields_ = [("evals", _I32), ("n_star", _I32), ("nonfinite", _I32), ("tr_extra_evals", _I32)]


class uad_kernel_stat(C.Structure):
    _fields_ = [("name", C.c_char * 32), ("launches", _I32), ("pad", _I32), ("total_ms", C.c_double),
                ("bytes", C.c_double), ("flops", C.c_double)]


def _fn(name, res, *args):
    f = getattr(_lib, name)
    f.restype = res
    f.argtypes = list(args)
    return f


uad_version = _fn("uad_version", C.c_char_p)
uad_last_error = _fn("uad_last_error", C.c_char_p, _P)
uad_init = _fn("uad_init", C.c_int, C.POINTER(uad_arch), _P, C.c_size_t, C.POINTER(_P))
uad_set_prefix_kv = _fn("uad_set_prefix_kv", C.c_int, _P, _I32, _P, _P, _I32, _I32)
uad_prepare_times = _fn("uad_prepare_times", C.c_int, _P, _I32)
uad_denoise = _fn("uad_denoise", C.c_int, _P, _P, C.POINTER(uad_schedule), _I32, _P)
uad_poll_released = _fn("uad_poll_released", C.c_int, _P, _I32, _I32, C.c_int64, _P, _P, _P)
uad_finish = _fn("uad_finish", C.c_int, _P, _P, _P, _P, C.POINTER(uad_stats), C.c_int64)
uad_step_times = _fn("uad_step_times", C.c_int, _P, _P, _I32)
uad_launches_per_chunk = _fn("uad_launches_per_chunk", C.c_int, _P, _I32, _I32)
uad_destroy = _fn("uad_destroy", None, _P)
uad_plan_step = _fn("uad_plan_step", C.c_int, _P, _I32, _I32, _I32, _P, _P, _P)
uad_profile_chunk = _fn("uad_profile_chunk", C.c_int, _P, _P, C.POINTER(uad_schedule), _P, _I32, C.c_int64)
uad_tile_weight = _fn("uad_tile_weight", C.c_int, _P, _I32, _I32, _P)
uad_linear = _fn("uad_linear", C.c_int, _P, _P, _P, _P, _I32, _I32, _I32, _P)
uad_linear_static_scratch = _fn("uad_linear_static_scratch", C.c_int, _P, _P, _P, _P, _I32, _I32, _I32, _P)
uad_set_wait_limit = _fn("uad_set_wait_limit", C.c_int, _P, C.c_int64, _I32)
uad_so3_check = _fn("uad_so3_check", C.c_int, _P, _I32, _P, _P)
UAD_ETOOBIG = -7

EXPORTS = ["uad_version", "uad_last_error", "uad_init", "uad_set_prefix_kv", "uad_prepare_times",
           "uad_denoise", "uad_poll_released", "uad_finish", "uad_step_times",
           "uad_launches_per_chunk", "uad_destroy", "uad_plan_step", "uad_profile_chunk",
           "uad_tile_weight", "uad_linear", "uad_linear_static_scratch", "uad_set_wait_limit",
           "uad_so3_check"]


def tile_weight(w):
    """fp32 [K][N] -> uint16 bf16 bits in the tensor-core projection layout (host only)."""
    w = np.ascontiguousarray(w, dtype=np.float32)
    K, N = w.shape
    out = np.empty(N * K, dtype=np.uint16)
    rc = uad_tile_weight(_ptr(w), K, N, _ptr(out))
    if rc:
        raise UADError(rc, "tile_weight: needs N % 128 == 0 and K % 64 == 0")
    return out


class UADError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"UAD error {code}: {msg}")
        self.code = code


def _ptr(a):
    """Raw address of a numpy array or torch tensor (contiguous), or None."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        if not a.flags["C_CONTIGUOUS"]:
            raise ValueError("buffer must be C-contiguous")
        return a.ctypes.data
    if not a.is_contiguous():
        raise ValueError("buffer must be contiguous")
    return a.data_ptr()


def _buf(a, n, dtype, what, host=False):
    """Address of a buffer the library reads or writes n elements of: a C-contiguous numpy
    array or torch tensor of `dtype` ("float32", "int32", "uint8"; "bfloat16" = np.uint16 bit
    patterns or a torch bfloat16 tensor) holding exactly n elements (host memory only when
    `host`). The C ABI takes bare pointers and cannot check sizes, so a short buffer is
    refused here, before the call, with ValueError; None passes through."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        ok = a.dtype == (np.dtype(np.uint16) if dtype == "bfloat16" else np.dtype(dtype))
        size, on_host = a.size, True
    else:
        ok = str(a.dtype) == "torch." + dtype
        size, on_host = a.numel(), a.device.type == "cpu"
    if not ok:
        raise ValueError(f"{what}: expected {dtype} elements, got {a.dtype}")
    if size != n:
        raise ValueError(f"{what}: expected {n} elements, got {size}")
    if host and not on_host:
        raise ValueError(f"{what}: must be host memory")
    return _ptr(a)


def _stream_handle(stream):
    if stream is None:
        return None
    return getattr(stream, "cuda_stream", stream)


def arch_struct(arch, max_batch=1):
    """uad_arch from any object with the architecture's attribute names."""
    g = (lambda k: arch[k]) if isinstance(arch, dict) else (lambda k: getattr(arch, k))
    kind, dt = g("kind"), g("dtype")
    return uad_arch(kind=KIND.get(kind, kind), dtype=DTYPE.get(dt, dt), n_layers=g("n_layers"),
                    width=g("width"), n_heads=g("n_heads"), n_kv_heads=g("n_kv_heads"),
                    head_dim=g("head_dim"), mlp_dim=g("mlp_dim"), action_dim=g("action_dim"),
                    chunk_len=g("chunk_len"), prefix_len=g("prefix_len"),
                    prefix_width=g("prefix_width"), rope=int(bool(g("rope"))), max_batch=max_batch)


def plan_step(budgets, k, tr=True):
    """Host-only plan of step k: (n_star, flags[H], tau_num[H], tau_den[H])."""
    b = np.ascontiguousarray(budgets, dtype=np.int32)
    H = b.size
    f, tn, td = (np.zeros(H, np.int32) for _ in range(3))
    ns = uad_plan_step(_ptr(b), H, k, int(tr), _ptr(f), _ptr(tn), _ptr(td))
    if ns < 0:
        raise UADError(ns, "invalid plan arguments")
    return ns, f, tn, td


class Expert:
    """One library context: an action expert's weights, prefixes and denoising state."""

    def __init__(self, arch, weights, max_batch=1):
        self.arch = arch_struct(arch, max_batch)
        self.H, self.D = self.arch.chunk_len, self.arch.action_dim
        h = _P()
        w = weights if not isinstance(weights, np.ndarray) else np.ascontiguousarray(weights, np.float32)
        n = w.size if isinstance(w, np.ndarray) else w.numel()
        rc = uad_init(C.byref(self.arch), _buf(w, n, "float32", "weights"), n, C.byref(h))
        if rc != UAD_OK:
            raise UADError(rc, "uad_init failed (see stderr)")
        self.h = h
        self._keep = None
        self._B = 1

    def _check(self, rc, what):
        if rc < 0:
            raise UADError(rc, f"{what}: {uad_last_error(self.h).decode()}")
        return rc

    def set_prefix(self, robot, k, v=None, dtype="f32"):
        """Attention-prefix experts: k, v [L][P][Hkv][dh]; DiT: k = prefix tokens
        [P][prefix_width], v = None. dtype "f32" (float32) or "bf16" (bfloat16 tensors or
        np.uint16 bit patterns); host or device."""
        code = DTYPE.get(dtype, dtype)
        el = "bfloat16" if code == DTYPE["bf16"] else "float32"
        a = self.arch
        if a.kind == KIND["dit"]:
            n = a.prefix_len * a.prefix_width
        else:
            n = a.n_layers * a.prefix_len * a.n_kv_heads * a.head_dim
        if isinstance(k, np.ndarray):
            k = np.ascontiguousarray(k, np.float32 if el == "float32" else None)
        if isinstance(v, np.ndarray):
            v = np.ascontiguousarray(v, np.float32 if el == "float32" else None)
        return self._check(uad_set_prefix_kv(self.h, robot, _buf(k, n, el, "prefix k"),
                                             _buf(v, n, el, "prefix v"), a.prefix_len, code),
                           "set_prefix")

    def prepare_times(self, max_budget):
        return self._check(uad_prepare_times(self.h, max_budget), "prepare_times")

    def _schedule(self, budgets, n_exec, tr, gac, chunk_relative, gac_mask, rot_dim=None):
        b = np.ascontiguousarray(budgets, dtype=np.int32).reshape(-1, self.H)
        m = None if gac_mask is None else np.ascontiguousarray(gac_mask, dtype=np.uint8)
        if m is not None and m.size != self.D:
            raise ValueError(f"gac_mask: expected {self.D} entries, got {m.size}")
        sc = uad_schedule(budgets=b.ctypes.data_as(C.POINTER(_I32)), batch=b.shape[0], n_exec=n_exec,
                          tr=int(tr), gac=int(gac), chunk_relative=int(chunk_relative),
                          gac_mask=None if m is None else m.ctypes.data_as(C.POINTER(C.c_uint8)),
                          rot_dim=-1 if rot_dim is None else int(rot_dim))
        return sc, (b, m)

    def denoise(self, noise, budgets, n_exec=0, tr=True, gac=True, chunk_relative=False,
                gac_mask=None, n_star=0, stream=None, rot_dim=None):
        """rot_dim: first of three rotation-vector dimensions corrected on SO(3) (None: none)."""
        sc, keep = self._schedule(budgets, n_exec, tr, gac, chunk_relative, gac_mask, rot_dim)
        if isinstance(noise, np.ndarray):
            noise = np.ascontiguousarray(noise, dtype=np.float32)
        B = keep[0].shape[0]
        p = _buf(noise, B * self.H * self.D, "float32", "noise")
        self._keep = noise
        self._B = B
        return self._check(uad_denoise(self.h, p, C.byref(sc), n_star, _stream_handle(stream)), "denoise")

    def profile(self, noise, budgets, n_exec=0, tr=True, gac=True, chunk_relative=False, gac_mask=None,
                timeout_us=120_000_000):
        """Per-kernel-class CUDA-event times of one eagerly launched chunk."""
        sc, keep = self._schedule(budgets, n_exec, tr, gac, chunk_relative, gac_mask)
        if isinstance(noise, np.ndarray):
            noise = np.ascontiguousarray(noise, dtype=np.float32)
        B = keep[0].shape[0]
        p = _buf(noise, B * self.H * self.D, "float32", "noise")
        self._B = B
        stats = (uad_kernel_stat * 64)()
        n = self._check(uad_profile_chunk(self.h, p, C.byref(sc), stats, 64, int(timeout_us)), "profile")
        return [dict(name=st.name.decode(), launches=st.launches, total_ms=st.total_ms, bytes=st.bytes,
                     flops=st.flops) for st in stats[:n]]

    def poll(self, robot, min_ready=1, timeout_us=0, out=None):
        out = np.zeros((self.H, self.D), np.float32) if out is None else out
        ready = np.zeros(self.H, np.int32)
        step = np.zeros(self.H, np.int32)
        p = _buf(out, self.H * self.D, "float32", "out", host=True)
        rc = uad_poll_released(self.h, robot, min_ready, int(timeout_us), p, _ptr(ready), _ptr(step))
        if rc < 0 and rc != UAD_ETIMEDOUT:
            self._check(rc, "poll")
        return rc, out, ready, step

    def finish(self, timeout_us=-1, final=None, ghost=None, gac_error=None, check=True):
        B = self._B
        final = np.zeros((B, self.H, self.D), np.float32) if final is None else final
        ghost = np.zeros((B, self.H, self.D), np.float32) if ghost is None else ghost
        gac_error = np.zeros((B, self.D), np.float32) if gac_error is None else gac_error
        st = uad_stats()
        n = B * self.H * self.D
        pf, pg = _buf(final, n, "float32", "final"), _buf(ghost, n, "float32", "ghost")
        pe = _buf(gac_error, B * self.D, "float32", "gac_error")
        rc = uad_finish(self.h, pf, pg, pe, C.byref(st), int(timeout_us))
        if check and rc < 0:
            self._check(rc, "finish")
        return dict(rc=rc, final=final, ghost=ghost, E=gac_error, evals=st.evals, n_star=st.n_star,
                    nonfinite=st.nonfinite, tr_extra_evals=st.tr_extra_evals)

    def step_times(self, n=MAX_STEPS):
        out = np.zeros(n, np.float64)
        k = self._check(uad_step_times(self.h, _ptr(out), n), "step_times")
        return out[:k]

    def set_wait_limit(self, wait_ns=2_000_000_000, unreachable=0):
        """Testing aid: bound of every wait in the persistent kernel, and extra arrivals its
        first completion count waits for (> 0: the wait runs out and the chunk reports an
        error)."""
        return self._check(uad_set_wait_limit(self.h, int(wait_ns), int(unreachable)), "set_wait_limit")

    def launches_per_chunk(self, batch, n_star):
        return self._check(uad_launches_per_chunk(self.h, batch, n_star), "launches")

    def close(self):
        if getattr(self, "h", None):
            uad_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
