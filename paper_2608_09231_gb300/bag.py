"""Python binding of the BAG C ABI (include/bag.h): argument marshalling only.

Every computation happens in libbag.so's CUDA kernels; this module converts configs to
the C structs, passes device pointers (torch tensors' data_ptr) and host buffers, and
turns status codes into exceptions.  It never falls back to anything: if the library is
missing or fails to load, load() raises.
"""

import ctypes
import os

import numpy as np

from . import configs as _configs

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libbag.so")

KIND = {"single": 0, "mmdit": 1, "wan": 2}
DTYPE = {"f32": 0, "bf16": 1}
GATE_KIND = {"mlp3": 0, "flux6": 1, "wan6": 2}
SAMPLER = {"euler": 0, "unipc": 1}
OBSERVABLE = {"modulated": 0, "embedded": 1}
POLICY_BAG, POLICY_FULL, POLICY_MASK, POLICY_STATIC_UNIFORM, POLICY_THRESHOLD = 0, 1, 2, 3, 4
LOG_FLOATS = 16
STATUS = {0: "BAG_OK", 1: "BAG_EINVAL", 2: "BAG_ENOMEM", 3: "BAG_ECUDA", 4: "BAG_EORDER",
          5: "BAG_EDEVICE_TIMEOUT", 6: "BAG_ESTATE", 7: "BAG_EUNSUPPORTED"}

EXPORTS = ["bag_create", "bag_destroy", "bag_last_error", "bag_set_stream", "bag_load_gate",
           "bag_set_policy", "bag_set_budget", "bag_reset", "bag_step", "bag_run", "bag_run_host",
           "bag_get_weight", "bag_forward_block", "bag_prepare", "bag_launch_count",
           "bag_gemm_bf16", "bag_attention_bf16", "bag_attention_f16", "bag_ln_mod", "bag_residual_add",
           "bag_profile_run", "bag_profile_launches", "bag_rel_l1", "bag_rel_l1_noalloc",
           "bag_check_wait_timeout"]

PROF_KINDS = ["gemm", "attention", "norm", "signal", "gate", "cache"]


class BagError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class Arch(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("hidden", ctypes.c_int), ("heads", ctypes.c_int),
                ("mlp", ctypes.c_int), ("n_double", ctypes.c_int), ("n_single", ctypes.c_int),
                ("n_wan", ctypes.c_int), ("grid", ctypes.c_int * 3), ("n_txt", ctypes.c_int),
                ("patch_ch", ctypes.c_int), ("rope_axes", ctypes.c_int * 3),
                ("dtype", ctypes.c_int), ("weight_seed", ctypes.c_uint64),
                ("gate_seed", ctypes.c_uint64), ("tau", ctypes.c_float),
                ("gate_kind", ctypes.c_int), ("cfg", ctypes.c_int), ("guidance", ctypes.c_float),
                ("qk_norm", ctypes.c_int), ("sampler", ctypes.c_int), ("shift", ctypes.c_float),
                ("observable", ctypes.c_int)]


class Cond(ctypes.Structure):
    _fields_ = [("txt", ctypes.c_void_p), ("pooled", ctypes.c_void_p),
                ("txt_uncond", ctypes.c_void_p), ("pooled_uncond", ctypes.c_void_p)]


class ProfEntry(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_long), ("ms", ctypes.c_double), ("flops", ctypes.c_double),
                ("bytes", ctypes.c_double)]


class ProfLaunch(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("m", ctypes.c_int), ("n", ctypes.c_int),
                ("k", ctypes.c_int), ("ms", ctypes.c_float), ("flops", ctypes.c_double),
                ("bytes", ctypes.c_double), ("variant", ctypes.c_int)]


class Stats(ctypes.Structure):
    _fields_ = [("mask", ctypes.POINTER(ctypes.c_uint8)), ("log", ctypes.POINTER(ctypes.c_float)),
                ("nfe", ctypes.c_int), ("T", ctypes.c_int), ("B", ctypes.c_int)]


_lib = None

_P = ctypes.c_void_p
_I = ctypes.c_int
_L = ctypes.c_long


def load(path=None):
    """Load libbag.so (raises if it is missing; no fallback path exists)."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    sig = {
        "bag_create": ([ctypes.POINTER(Arch), _I, _I, ctypes.POINTER(_P)], _I),
        "bag_destroy": ([_P], None),
        "bag_last_error": ([_P], ctypes.c_char_p),
        "bag_set_stream": ([_P, _P], _I),
        "bag_load_gate": ([_P, _P, _I, _P, _P], _I),
        "bag_set_policy": ([_P, _I, _P, ctypes.c_float], _I),
        "bag_set_budget": ([_P, _I], _I),
        "bag_check_wait_timeout": ([_P], _I),
        "bag_reset": ([_P], _I),
        "bag_step": ([_P, _P, _I, ctypes.POINTER(Cond), _P, _P], _I),
        "bag_run": ([_P, _P, ctypes.POINTER(Cond), ctypes.POINTER(Stats)], _I),
        "bag_run_host": ([_P, _P, ctypes.POINTER(Cond), ctypes.POINTER(Stats)], _I),
        "bag_get_weight": ([_P, _I, ctypes.c_char_p, _P, ctypes.c_size_t], _I),
        "bag_forward_block": ([_P, _I, _I, _P], _I),
        "bag_prepare": ([_P, ctypes.POINTER(Cond)], _I),
        "bag_launch_count": ([_P, ctypes.POINTER(_L)], _I),
        "bag_gemm_bf16": ([_P, _P, _L, _P, _L, _P, _P, _L, _I, _I, _I, _I, _I], _I),
        "bag_attention_bf16": ([_P, _P, _P, _P, _P, _L, _I, _I, _I, _I, _L, _I], _I),
        "bag_attention_f16": ([_P, _P, _P, _P, _P, _L, _I, _I, _I, _I, _L], _I),
        "bag_ln_mod": ([_P, _P, _P, _P, _P, _I, _I], _I),
        "bag_residual_add": ([_P, _P, _P, _P, _L], _I),
        "bag_rel_l1": ([_P, _P, _P, _I, _L, _L, _P, _P], _I),
        "bag_rel_l1_noalloc": ([_P, _P, _I, _L, _L, _P, _P], _I),
        "bag_profile_run": ([_P, _P, ctypes.POINTER(Cond), ctypes.POINTER(Stats),
                             ctypes.POINTER(ProfEntry)], _I),
        "bag_profile_launches": ([_P, ctypes.POINTER(ProfLaunch), _L, ctypes.POINTER(_L)], _I),
    }
    for name, (args, res) in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    _lib = lib
    return lib


def arch_from_config(cfg, tau=0.5):
    a = Arch()
    a.kind = KIND[cfg["kind"]]
    a.hidden, a.heads, a.mlp = cfg["hidden"], cfg["heads"], cfg["mlp"]
    a.n_double, a.n_single, a.n_wan = cfg["n_double"], cfg["n_single"], cfg["n_wan"]
    a.grid[:] = list(cfg["grid"])
    a.n_txt, a.patch_ch = cfg["n_txt"], cfg["patch_ch"]
    a.rope_axes[:] = list(cfg["rope_axes"])
    a.dtype = DTYPE[cfg["dtype"]]
    a.weight_seed, a.gate_seed = cfg["weight_seed"], cfg["gate_seed"]
    a.tau = tau
    a.gate_kind = GATE_KIND[cfg.get("gate_kind", "mlp3")]
    g = cfg.get("guidance")
    a.cfg = 0 if g is None else 1
    a.guidance = 0.0 if g is None else float(g)
    a.qk_norm = 1 if cfg.get("qk_norm") else 0
    a.sampler = SAMPLER[cfg.get("sampler", "euler")]
    a.shift = float(cfg.get("shift", 1.0))
    a.observable = OBSERVABLE[cfg.get("observable", "modulated")]
    return a


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _dp(t):
    return None if t is None else t.data_ptr()


def _cond(txt, pooled, txt_u=None, pooled_u=None):
    """Device conditioning (torch tensors; the *_u pair is the unconditional branch of
    a guided context)."""
    return Cond(_dp(txt), _dp(pooled), _dp(txt_u), _dp(pooled_u))


class Context:
    """A bag_ctx: one model instance, one sample at a time (bag_create ... bag_destroy)."""

    def __init__(self, cfg, T=None, B=None, tau=0.5):
        self.lib = load()
        self.cfg = cfg
        self.T = cfg["T"] if T is None else T
        self.B = cfg["budgets"][0] if B is None else B
        self._arch = arch_from_config(cfg, tau)
        h = ctypes.c_void_p()
        st = self.lib.bag_create(ctypes.byref(self._arch), self.T, self.B, ctypes.byref(h))
        if st != 0:
            raise BagError(st, self.lib.bag_last_error(None).decode())
        self.h = h

    def _chk(self, st):
        if st != 0:
            raise BagError(st, self.lib.bag_last_error(self.h).decode())

    def close(self):
        if getattr(self, "h", None):
            self.lib.bag_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # --- API mirror -----------------------------------------------------------------
    def set_stream(self, stream):
        self._chk(self.lib.bag_set_stream(self.h, ctypes.c_void_p(stream)))

    def load_gate(self, theta, mu=None, sd=None):
        th = np.ascontiguousarray(theta, np.float32)
        mu_a = None if mu is None else np.ascontiguousarray(mu, np.float32)
        sd_a = None if sd is None else np.ascontiguousarray(sd, np.float32)
        self._chk(self.lib.bag_load_gate(self.h, th.ctypes.data, th.size,
                                         None if mu_a is None else mu_a.ctypes.data,
                                         None if sd_a is None else sd_a.ctypes.data))

    def set_policy(self, policy, mask=None, delta=0.0):
        m = None if mask is None else np.ascontiguousarray(mask, np.uint8)
        self._chk(self.lib.bag_set_policy(self.h, policy, None if m is None else m.ctypes.data,
                                          float(delta)))

    def set_budget(self, B):
        """Budget of later samples (the step graph is re-captured on the next run)."""
        self._chk(self.lib.bag_set_budget(self.h, int(B)))
        self.B = int(B)

    def reset(self):
        self._chk(self.lib.bag_reset(self.h))

    def check_wait_timeout(self):
        """bag_check_wait_timeout: returns the status (BAG_EDEVICE_TIMEOUT expected)."""
        return self.lib.bag_check_wait_timeout(self.h)

    def prepare(self, txt, pooled, txt_u=None, pooled_u=None):
        c = _cond(txt, pooled, txt_u, pooled_u)
        self._chk(self.lib.bag_prepare(self.h, ctypes.byref(c)))

    def step(self, x, t, txt, pooled, x_out, flag=None, txt_u=None, pooled_u=None):
        c = _cond(txt, pooled, txt_u, pooled_u)
        self._chk(self.lib.bag_step(self.h, _ptr(x), t, ctypes.byref(c), _ptr(x_out), _ptr(flag)))

    def _stats(self):
        mask = np.zeros(self.T, np.uint8)
        log = np.zeros((self.T, LOG_FLOATS), np.float32)
        s = Stats(mask.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)),
                  log.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), 0, 0, 0)
        return s, mask, log

    def run(self, x, txt, pooled, txt_u=None, pooled_u=None):
        """All T steps in place on device tensor x; returns (mask, log, nfe)."""
        c = _cond(txt, pooled, txt_u, pooled_u)
        s, mask, log = self._stats()
        self._chk(self.lib.bag_run(self.h, _ptr(x), ctypes.byref(c), ctypes.byref(s)))
        return mask, log, s.nfe

    def profile_run(self, x, txt, pooled, txt_u=None, pooled_u=None):
        """Profiled sample (direct launches with events); returns (mask, log, nfe, prof)
        where prof maps a kernel class to dict(launches, ms, flops, bytes)."""
        c = _cond(txt, pooled, txt_u, pooled_u)
        s, mask, log = self._stats()
        out = (ProfEntry * len(PROF_KINDS))()
        self._chk(self.lib.bag_profile_run(self.h, _ptr(x), ctypes.byref(c), ctypes.byref(s), out))
        prof = {k: dict(launches=out[i].launches, ms=out[i].ms, flops=out[i].flops,
                        bytes=out[i].bytes) for i, k in enumerate(PROF_KINDS)}
        return mask, log, s.nfe, prof

    def profile_launches(self):
        """Per-launch records of the last profile_run as a list of dicts."""
        n = ctypes.c_long()
        self._chk(self.lib.bag_profile_launches(self.h, None, 0, ctypes.byref(n)))
        arr = (ProfLaunch * max(1, n.value))()
        self._chk(self.lib.bag_profile_launches(self.h, arr, n.value, ctypes.byref(n)))
        return [dict(kind=PROF_KINDS[r.kind], m=r.m, n=r.n, k=r.k, ms=r.ms, flops=r.flops,
                     bytes=r.bytes, variant=r.variant) for r in arr[:n.value]]

    def run_host(self, x, txt, pooled, txt_u=None, pooled_u=None):
        """All T steps with host numpy buffers (x updated in place); returns (mask, log, nfe)."""
        assert x.dtype == np.float32 and x.flags.c_contiguous
        keep = [None if a is None else np.ascontiguousarray(a, np.float32)
                for a in (txt, pooled, txt_u, pooled_u)]
        c = Cond(*[None if a is None else a.ctypes.data for a in keep])
        s, mask, log = self._stats()
        self._chk(self.lib.bag_run_host(self.h, x.ctypes.data, ctypes.byref(c), ctypes.byref(s)))
        return mask, log, s.nfe

    def get_weight(self, block, name, n):
        out = np.empty(n, np.float32)
        self._chk(self.lib.bag_get_weight(self.h, block, name.encode(), out.ctypes.data, n))
        return out

    def forward_block(self, block, t_mod, h):
        self._chk(self.lib.bag_forward_block(self.h, block, t_mod, _ptr(h)))

    def launch_count(self):
        n = ctypes.c_long()
        self._chk(self.lib.bag_launch_count(self.h, ctypes.byref(n)))
        return n.value

    def gemm_bf16(self, A, W, bias, C, M, N, K, epilogue=0, force_simt=0):
        self._chk(self.lib.bag_gemm_bf16(self.h, _ptr(A), A.stride(0), _ptr(W), W.stride(0),
                                         _ptr(bias), _ptr(C), C.stride(0), M, N, K, epilogue,
                                         force_simt))

    def attention_bf16(self, q, k, v, o, nq, nk, heads, dh, vpad=0, force_simt=0):
        """v: [nk, ld] when vpad == 0, else transposed per head [heads, dh, vpad]."""
        self._chk(self.lib.bag_attention_bf16(self.h, _ptr(q), _ptr(k), _ptr(v), _ptr(o),
                                              q.stride(0), nq, nk, heads, dh, vpad, force_simt))

    def attention_f16(self, q, k, v, o, nq, nk, heads, dh, vpad):
        """fp16 q, k and v (v transposed per head, [heads, dh, vpad]); bf16 output."""
        self._chk(self.lib.bag_attention_f16(self.h, _ptr(q), _ptr(k), _ptr(v), _ptr(o),
                                             q.stride(0), nq, nk, heads, dh, vpad))

    def ln_mod(self, x, shift, scale, y, rows, cols):
        self._chk(self.lib.bag_ln_mod(self.h, _ptr(x), _ptr(shift), _ptr(scale), _ptr(y), rows,
                                      cols))

    def rel_l1(self, a, b, rows, cols, scratch, out, bf16=None):
        dt = (1 if a.dtype.itemsize == 2 else 0) if bf16 is None else int(bf16)
        self._chk(self.lib.bag_rel_l1(self.h, _ptr(a), _ptr(b), dt, rows, cols, _ptr(scratch),
                                      _ptr(out)))

    def residual_add(self, out, h_in, R, n):
        self._chk(self.lib.bag_residual_add(self.h, _ptr(out), _ptr(h_in), _ptr(R), n))


def rel_l1_noalloc(a, b, rows, cols, out, stream=0, bf16=None):
    """bag_rel_l1_noalloc: the signal reduction with no context and no allocation
    (scratch in a fixed device array of the library; see include/bag.h)."""
    lib = load()
    dt = (1 if a.dtype.itemsize == 2 else 0) if bf16 is None else int(bf16)
    st = lib.bag_rel_l1_noalloc(_ptr(a), _ptr(b), dt, rows, cols, _ptr(out),
                                ctypes.c_void_p(stream))
    if st != 0:
        raise BagError(st, lib.bag_last_error(None).decode())


def create(cfg_or_name, T=None, B=None, tau=0.5, **overrides):
    cfg = (_configs.get_config(cfg_or_name, **overrides) if isinstance(cfg_or_name, str)
           else cfg_or_name)
    return Context(cfg, T=T, B=B, tau=tau)
