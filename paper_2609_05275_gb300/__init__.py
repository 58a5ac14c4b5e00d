"""Python binding of libld.so, the sm_103a layer-dropout decoder-stack library.

Argument marshalling only: every step of the forward and backward pass runs in
the library's CUDA kernels behind the C ABI of ``include/ld.h``.  PyTorch
provides device memory and the current stream.  There is no fallback: if
``libld.so`` has not been built, every call raises.

Functions keep the C names (``ld_create``, ``ld_set_schedule``,
``ld_forward``, ``ld_backward``, ...); ``LayerDropStack`` bundles a handle,
its workspace and the per-layer pointer tables for convenience.
"""

import ctypes
import os
import re

from ctypes import POINTER, c_char_p, c_double, c_float, c_int, c_longlong, c_size_t, c_ulonglong, c_void_p

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libld.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "ld.h")

# enums of include/ld.h
LD_OK, LD_ERR_ARG, LD_ERR_SHAPE, LD_ERR_STATE, LD_ERR_CUDA, LD_ERR_TIMEOUT, LD_ERR_OOM, LD_ERR_UNSUPPORTED = range(8)
LD_PER_SEQUENCE, LD_PER_BATCH, LD_PER_SHARD, LD_PER_TOKEN = 0, 1, 2, 3
LD_DIST_UNIFORM, LD_DIST_ILD, LD_DIST_ALD, LD_DIST_EXPLICIT = 0, 1, 2, 3
LD_TIME_CONST, LD_TIME_ITS, LD_TIME_DTS, LD_TIME_RAMP = 0, 1, 2, 3
DIST = {"uniform": LD_DIST_UNIFORM, "ild": LD_DIST_ILD, "ald": LD_DIST_ALD, "explicit": LD_DIST_EXPLICIT}
TIME = {"const": LD_TIME_CONST, "its": LD_TIME_ITS, "dts": LD_TIME_DTS, "ramp": LD_TIME_RAMP}
ACT = {"swiglu": 0, "relu2": 1}
GRAN = {"per_sequence": LD_PER_SEQUENCE, "per_batch": LD_PER_BATCH, "per_shard": LD_PER_SHARD,
        "per_token": LD_PER_TOKEN}


class ld_config(ctypes.Structure):
    _fields_ = [("L", c_int), ("d", c_int), ("H", c_int), ("Hkv", c_int), ("Dh", c_int), ("F", c_int),
                ("B", c_int), ("S", c_int), ("eps", c_float), ("rope_theta", c_float), ("alpha", c_float),
                ("granularity", c_int), ("fp32_debug", c_int), ("b_offset", c_int), ("sublayer", c_int),
                ("alibi", c_int), ("act", c_int)]


class ld_schedule(ctypes.Structure):
    _fields_ = [("dist", c_int), ("p_max", c_float), ("p_explicit", POINTER(c_float)), ("time", c_int),
                ("T", c_longlong), ("ramp_t0", c_longlong), ("ramp_t1", c_longlong), ("ramp_s0", c_float),
                ("ramp_s1", c_float), ("seed", c_ulonglong)]


_WNAMES = ("w_qkv", "w_o", "w_gu", "w_d", "g1", "g2")


class ld_layer_w(ctypes.Structure):
    _fields_ = [(n, c_void_p) for n in _WNAMES]


class ld_layer_g(ctypes.Structure):
    _fields_ = [(n, c_void_p) for n in _WNAMES]


class LdError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        msg = f"{where}: {ld_status_str(status)} (status {status})"
        if status == LD_ERR_CUDA:
            msg += ": " + lib().ld_last_cuda_error().decode()
        super().__init__(msg)


_lib = None


def lib():
    """Load libld.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2609_05275_gb300.build.build()")
        import torch  # noqa: F401  (loads the CUDA runtime the library links against)
        L = ctypes.CDLL(LIB_PATH)
        sigs = {
            "ld_create": (c_int, [POINTER(ld_config), POINTER(c_void_p)]),
            "ld_workspace_size": (c_int, [c_void_p, POINTER(c_size_t)]),
            "ld_set_schedule": (c_int, [c_void_p, POINTER(ld_schedule)]),
            "ld_get_rates": (c_int, [c_void_p, c_longlong, POINTER(c_double), POINTER(c_ulonglong), POINTER(c_float)]),
            "ld_draw_masks": (c_int, [c_void_p, c_longlong, c_void_p, c_void_p]),
            "ld_forward": (c_int, [c_void_p, c_longlong, POINTER(ld_layer_w), c_void_p, c_void_p, c_void_p]),
            "ld_backward": (c_int, [c_void_p, POINTER(ld_layer_w), c_void_p, POINTER(ld_layer_g), c_void_p, c_void_p]),
            "ld_forward_eval": (c_int, [c_void_p, c_void_p, c_void_p, POINTER(ld_layer_w), c_void_p, c_void_p,
                                        c_void_p]),
            "ld_eval_workspace_size": (c_int, [c_void_p, POINTER(c_size_t)]),
            "ld_get_masks": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p]),
            "ld_sync": (c_int, [c_void_p]),
            "ld_destroy": (c_int, [c_void_p]),
            "ld_status_str": (c_char_p, [c_int]),
            "ld_last_cuda_error": (c_char_p, []),
            "ld_set_timing": (c_int, [c_void_p, c_int]),
            "ld_get_timing": (c_int, [c_void_p, c_int, POINTER(c_double), POINTER(c_longlong)]),
            "ld_rmsnorm_backward": (c_int, [c_int, c_int, c_int, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                            c_void_p, c_void_p, c_void_p, c_float, c_void_p, c_void_p, c_size_t,
                                            c_void_p]),
            "ld_rmsnorm_backward_noalloc": (c_int, [c_int, c_int, c_int, c_void_p, c_void_p, c_void_p, c_void_p,
                                                    c_void_p, c_void_p, c_void_p, c_void_p, c_float, c_void_p,
                                                    c_void_p]),
            "ld_gemm_bf16": (c_int, [c_int, c_int, c_int, c_void_p, c_int, c_int, c_void_p, c_int, c_int, c_void_p,
                                     c_int, c_int, c_float, c_void_p, c_void_p]),
            "ld_check_wait_timeout": (c_int, [c_void_p, c_void_p]),
        }
        for name, (res, args) in sigs.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def header_functions():
    """Names of the functions include/ld.h declares."""
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(ld_\w+)\s*\(", src, flags=re.M)))


def _check(status, where):
    if status != LD_OK:
        raise LdError(status, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


# --------------------------------------------------------------- C functions
def ld_status_str(status):
    return lib().ld_status_str(int(status)).decode()


def make_config(cfg, granularity="per_sequence", fp32_debug=False, b_offset=0, sublayer=False):
    return ld_config(cfg["L"], cfg["d"], cfg["H"], cfg["Hkv"], cfg["Dh"], cfg["F"], cfg["B"], cfg["S"],
                     cfg.get("eps", 1e-6), cfg.get("rope_theta", 0.0), cfg.get("alpha", 1.0),
                     GRAN[granularity] if isinstance(granularity, str) else int(granularity), int(fp32_debug),
                     int(b_offset), int(sublayer), int(bool(cfg.get("alibi", False))),
                     ACT[cfg.get("act", "swiglu")])


def ld_create(config):
    h = c_void_p()
    _check(lib().ld_create(ctypes.byref(config), ctypes.byref(h)), "ld_create")
    return h


def ld_create_status(config):
    """Status code of ld_create (for argument-validation tests); destroys the handle."""
    h = c_void_p()
    st = lib().ld_create(ctypes.byref(config), ctypes.byref(h))
    if st == LD_OK:
        lib().ld_destroy(h)
    return st


def ld_workspace_size(h):
    n = c_size_t()
    _check(lib().ld_workspace_size(h, ctypes.byref(n)), "ld_workspace_size")
    return n.value


def make_schedule(sched):
    pe = sched.get("p_explicit")
    arr = (c_float * len(pe))(*pe) if pe is not None else None
    ramp = sched.get("ramp", (0, 1, 0.0, 1.0))
    s = ld_schedule(DIST[sched["dist"]], sched.get("p_max", 0.0), ctypes.cast(arr, POINTER(c_float)) if arr else None,
                    TIME[sched.get("time", "const")], sched.get("T", 0) or 0, ramp[0], ramp[1], ramp[2], ramp[3],
                    sched.get("seed", 0))
    s._keep = arr
    return s


def ld_set_schedule(h, schedule):
    st = lib().ld_set_schedule(h, ctypes.byref(schedule))
    _check(st, "ld_set_schedule")


def ld_set_schedule_status(h, schedule):
    return lib().ld_set_schedule(h, ctypes.byref(schedule))


def ld_get_rates(h, step, L):
    p = (c_double * L)()
    thr = (c_ulonglong * L)()
    sc = (c_float * L)()
    _check(lib().ld_get_rates(h, step, p, thr, sc), "ld_get_rates")
    return list(p), list(thr), list(sc)


def ld_draw_masks(h, step, workspace, stream=None):
    _check(lib().ld_draw_masks(h, step, _ptr(workspace), _stream(stream)), "ld_draw_masks")


def ld_forward(h, step, wtab, x, workspace, stream=None):
    _check(lib().ld_forward(h, step, wtab, _ptr(x), _ptr(workspace), _stream(stream)), "ld_forward")


def ld_backward(h, wtab, dx, gtab, workspace, stream=None):
    _check(lib().ld_backward(h, wtab, _ptr(dx), gtab, _ptr(workspace), _stream(stream)), "ld_backward")


def ld_eval_workspace_size(h):
    n = c_size_t()
    _check(lib().ld_eval_workspace_size(h, ctypes.byref(n)), "ld_eval_workspace_size")
    return n.value


def ld_forward_eval(h, execute, r_eval, wtab, x, workspace, stream=None):
    """execute: sequence of L 0/1 flags; r_eval: sequence of L floats or None."""
    import numpy as np
    ex = np.ascontiguousarray(np.asarray(execute, dtype=np.uint8))
    rv = None if r_eval is None else np.ascontiguousarray(np.asarray(r_eval, dtype=np.float32))
    _check(lib().ld_forward_eval(h, ex.ctypes.data, None if rv is None else rv.ctypes.data, wtab, _ptr(x),
                                 _ptr(workspace), _stream(stream)), "ld_forward_eval")


def ld_get_masks(h, L, B, sublayer=False, S=None):
    """(mask, kept_idx, kept_cnt) as [L, B], [L, B], [L]; with sub-layer
    granularity [2, L, B], [2, L, B], [2, L] (attention, then FFN).  Per
    token (pass S): mask [L, B, S], kept_idx [L, B*S] (kept token rows), and
    the kept-token counts [L] (leading axis 2 with sub-layer granularity)."""
    import numpy as np
    nm = 2 if sublayer else 1
    per = B * S if S else B
    mask = np.zeros(nm * L * per, dtype=np.uint8)
    idx = np.zeros(nm * L * per, dtype=np.int32)
    cnt = np.zeros(nm * L, dtype=np.int32)
    _check(lib().ld_get_masks(h, mask.ctypes.data, idx.ctypes.data, cnt.ctypes.data), "ld_get_masks")
    mshape = (L, B, S) if S else (L, B)
    if sublayer:
        return mask.reshape((2,) + mshape), idx.reshape(2, L, per), cnt.reshape(2, L)
    return mask.reshape(mshape), idx.reshape(L, per), cnt


def ld_sync(h):
    return lib().ld_sync(h)


def ld_destroy(h):
    _check(lib().ld_destroy(h), "ld_destroy")


LD_KCLASS_GEMM, LD_KCLASS_ATTN, LD_KCLASS_ROWWISE = 0, 1, 2


def ld_set_timing(h, enable):
    _check(lib().ld_set_timing(h, int(enable)), "ld_set_timing")


def ld_get_timing(h, kclass):
    ms = c_double()
    n = c_longlong()
    _check(lib().ld_get_timing(h, kclass, ctypes.byref(ms), ctypes.byref(n)), "ld_get_timing")
    return ms.value, n.value


def ld_gemm_bf16(M, N, K, A, lda, a_mn, B, ldb, b_mn, D, ldd, alpha=1.0, status=None, stream=None):
    import torch
    d_f32 = 1 if D.dtype == torch.float32 else 0
    _check(lib().ld_gemm_bf16(M, N, K, _ptr(A), lda, int(a_mn), _ptr(B), ldb, int(b_mn), _ptr(D), ldd, d_f32,
                              float(alpha), _ptr(status), _stream(stream)), "ld_gemm_bf16")


def ld_check_wait_timeout(status, stream=None):
    """Launch the bounded-wait failure-path check (include/ld.h); `status`
    is an int32 device tensor of one element."""
    _check(lib().ld_check_wait_timeout(_ptr(status), _stream(stream)), "ld_check_wait_timeout")


def rmsnorm_backward_scratch_bytes(B, S, d):
    nb = min((B * S + 7) // 8, 320)
    return nb * d * 4


def ld_rmsnorm_backward(B, S, d, dyn, xs, rstd, gamma, kept_idx, kept_cnt, dx, nxt, scale, dgamma, scratch,
                        stream=None):
    _check(lib().ld_rmsnorm_backward(B, S, d, _ptr(dyn), _ptr(xs), _ptr(rstd), _ptr(gamma), _ptr(kept_idx),
                                     _ptr(kept_cnt), _ptr(dx), _ptr(nxt), float(scale), _ptr(dgamma), _ptr(scratch),
                                     scratch.numel() * scratch.element_size(), _stream(stream)),
           "ld_rmsnorm_backward")


def ld_rmsnorm_backward_noalloc(B, S, d, dyn, xs, rstd, gamma, kept_idx, kept_cnt, dx, nxt, scale, dgamma,
                                stream=None):
    _check(lib().ld_rmsnorm_backward_noalloc(B, S, d, _ptr(dyn), _ptr(xs), _ptr(rstd), _ptr(gamma), _ptr(kept_idx),
                                             _ptr(kept_cnt), _ptr(dx), _ptr(nxt), float(scale), _ptr(dgamma),
                                             _stream(stream)),
           "ld_rmsnorm_backward_noalloc")


def weight_table(layers):
    """ld_layer_w[L] from a list of dicts of device tensors (None: a layer
    whose weights are never read, e.g. one skipped by ld_forward_eval)."""
    tab = (ld_layer_w * len(layers))()
    for i, W in enumerate(layers):
        if W is None:
            continue
        for n in _WNAMES:
            setattr(tab[i], n, W[n].data_ptr())
    tab._keep = layers
    return tab


def grad_table(grads):
    tab = (ld_layer_g * len(grads))()
    for i, G in enumerate(grads):
        for n in _WNAMES:
            setattr(tab[i], n, G[n].data_ptr())
    tab._keep = grads
    return tab


class LayerDropStack:
    """A handle with its workspace: forward / backward of the whole stack."""

    def __init__(self, cfg, sched, granularity="per_sequence", fp32_debug=False, device="cuda", b_offset=0,
                 sublayer=False):
        import torch
        self.cfg = dict(cfg)
        self.sublayer = bool(sublayer)
        self.per_token = granularity == "per_token" or granularity == LD_PER_TOKEN
        self.config = make_config(cfg, granularity, fp32_debug, b_offset, sublayer)
        self.h = ld_create(self.config)
        self.schedule = make_schedule(sched)
        ld_set_schedule(self.h, self.schedule)
        nbytes = ld_workspace_size(self.h)
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=device)
        self.dtype = torch.float32 if fp32_debug else torch.bfloat16

    def rates(self, step):
        return ld_get_rates(self.h, step, self.cfg["L"])

    def draw_masks(self, step, stream=None):
        ld_draw_masks(self.h, step, self.workspace, stream)
        return self.masks()

    def masks(self):
        return ld_get_masks(self.h, self.cfg["L"], self.cfg["B"], self.sublayer,
                            self.cfg["S"] if self.per_token else None)

    def forward(self, step, wtab, x, stream=None):
        ld_forward(self.h, step, wtab, x, self.workspace, stream)

    def backward(self, wtab, dx, gtab, stream=None):
        ld_backward(self.h, wtab, dx, gtab, self.workspace, stream)

    def forward_eval(self, execute, wtab, x, r_eval=None, stream=None):
        """Inference forward on the executed layers (in place on x)."""
        ld_forward_eval(self.h, execute, r_eval, wtab, x, self.workspace, stream)

    def sync(self):
        st = ld_sync(self.h)
        _check(st, "ld_sync")

    def close(self):
        if self.h is not None:
            ld_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
