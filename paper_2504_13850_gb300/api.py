"""ctypes binding of the C ABI in include/fedoptima.h (argument marshalling
only: every step of the hot path runs in the library's CUDA kernels).

Buffers may be numpy arrays (host) or torch tensors (host, pinned or on the
GPU); they are passed by address.  Loading fails loudly when the library has
not been built: there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libfedoptima.so")

OK, EMPTY, FULL, STALE = 0, 1, 2, 3
ERR_ARG, ERR_CUDA, ERR_OOM, ERR_TIMEOUT, ERR_UNSUPPORTED = -1, -2, -3, -4, -5
STATUS = {0: "OK", 1: "EMPTY", 2: "FULL", 3: "STALE", -1: "ERR_ARG", -2: "ERR_CUDA",
          -3: "ERR_OOM", -4: "ERR_TIMEOUT", -5: "ERR_UNSUPPORTED"}

OP_KINDS = {"conv": 1, "affine": 2, "relu": 3, "maxpool2": 4, "add": 5, "avgpool": 6,
            "flatten": 7, "linear": 8, "layernorm": 9, "gelu": 10, "attention": 11,
            "meanpool": 12, "dwconv": 13, "hswish": 14, "hsigmoid": 15, "chmul": 16}
DTYPE_F32, DTYPE_BF16 = 0, 1
SCHED_COUNTER, SCHED_FIFO = 0, 1


class fo_op(C.Structure):
    _fields_ = [(n, C.c_int32) for n in
                ("kind", "in0", "in1", "cin", "cout", "k", "stride", "bias", "heads")]


class fo_optimizer(C.Structure):
    _fields_ = [("lr", C.c_float), ("momentum", C.c_float)]


class fo_server_cfg(C.Structure):
    _fields_ = [(n, C.c_int32) for n in
                ("num_devices", "omega", "depth", "batch", "in_h", "in_w", "in_c",
                 "num_classes", "dtype", "seq", "max_delay", "sched_policy")]


class FedOptimaError(RuntimeError):
    pass


_lib = None

# (name, restype, argtypes)
_SIGS = [
    ("fo_server_create", C.c_int, [C.POINTER(fo_op), C.c_int, C.POINTER(fo_optimizer),
                                   C.POINTER(fo_server_cfg), C.POINTER(C.c_void_p)]),
    ("fo_server_destroy", C.c_int, [C.c_void_p]),
    ("fo_server_num_params", C.c_int64, [C.c_void_p]),
    ("fo_server_set_params", C.c_int, [C.c_void_p, C.c_void_p, C.c_int64]),
    ("fo_server_get_params", C.c_int, [C.c_void_p, C.c_void_p, C.c_int64]),
    ("fo_server_set_momentum", C.c_int, [C.c_void_p, C.c_void_p, C.c_int64]),
    ("fo_server_get_momentum", C.c_int, [C.c_void_p, C.c_void_p, C.c_int64]),
    ("fo_enqueue_activations", C.c_int, [C.c_void_p, C.c_int, C.c_void_p, C.c_void_p,
                                         C.c_void_p, C.POINTER(C.c_int)]),
    ("fo_server_step", C.c_int, [C.c_void_p, C.POINTER(C.c_int), C.POINTER(C.c_int32)]),
    ("fo_read_losses", C.c_int, [C.c_void_p, C.c_void_p, C.c_int64, C.c_int64]),
    ("fo_aggregate", C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int64, C.c_int,
                               C.c_int32, C.POINTER(C.c_int32)]),
    ("fo_get_counters", C.c_int, [C.c_void_p, C.c_void_p]),
    ("fo_get_sender_status", C.c_int, [C.c_void_p, C.c_void_p]),
    ("fo_get_version", C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.POINTER(C.c_int32)]),
    ("fo_set_device_active", C.c_int, [C.c_void_p, C.c_int, C.c_int]),
    ("fo_server_activation_bytes", C.c_int64, [C.c_void_p]),
    ("fo_server_synchronize", C.c_int, [C.c_void_p]),
    ("fo_server_stream", C.c_void_p, [C.c_void_p]),
    ("fo_server_agg_stream", C.c_void_p, [C.c_void_p]),
    ("fo_server_join_aggregations", C.c_int, [C.c_void_p]),
    ("fo_server_last_step_launches", C.c_int, [C.c_void_p]),
    ("fo_server_profile", C.c_int, [C.c_void_p, C.c_int]),
    ("fo_server_kernel_times", C.c_int, [C.c_void_p, C.POINTER(C.c_char_p), C.POINTER(C.c_int64),
                                         C.POINTER(C.c_double), C.POINTER(C.c_double),
                                         C.POINTER(C.c_double), C.c_int, C.POINTER(C.c_int)]),
    ("fo_server_profile_reset", C.c_int, [C.c_void_p]),
    ("fo_server_kernels_launched", C.c_int64, [C.c_void_p]),
    ("fo_server_device_bytes", C.c_int64, [C.c_void_p]),
    ("fo_server_error", C.c_int, [C.c_void_p]),
    ("fo_last_error", C.c_char_p, []),
    ("fo_sched_create", C.c_int, [C.c_int, C.c_int, C.c_int, C.c_int, C.POINTER(C.c_void_p)]),
    ("fo_sched_destroy", C.c_int, [C.c_void_p]),
    ("fo_sched_put", C.c_int, [C.c_void_p, C.c_int, C.POINTER(C.c_int32), C.POINTER(C.c_int)]),
    ("fo_sched_get", C.c_int, [C.c_void_p, C.POINTER(C.c_int), C.POINTER(C.c_int32)]),
    ("fo_sched_set_active", C.c_int, [C.c_void_p, C.c_int, C.c_int]),
    ("fo_sched_counters", C.c_int, [C.c_void_p, C.c_void_p]),
    ("fo_sched_sender_status", C.c_int, [C.c_void_p, C.c_void_p]),
    ("fo_sched_queued", C.c_int, [C.c_void_p, C.c_int]),
    ("fo_axpby_async", C.c_int, [C.c_void_p, C.c_void_p, C.c_int64, C.c_float, C.c_void_p]),
    ("fo_column_sums", C.c_int, [C.c_void_p, C.c_int, C.c_int64, C.c_int, C.c_void_p, C.c_void_p]),
    ("fo_column_sums_noalloc", C.c_int, [C.c_void_p, C.c_int, C.c_int64, C.c_int, C.c_void_p, C.c_void_p]),
    ("fo_server_tensor", C.c_int, [C.c_void_p, C.c_int, C.POINTER(C.c_void_p), C.POINTER(C.c_int64),
                                   C.POINTER(C.c_int)]),
    ("fo_server_params_device", C.c_int, [C.c_void_p, C.POINTER(C.c_void_p), C.POINTER(C.c_int64)]),
    ("fo_server_load_params_device", C.c_int, [C.c_void_p, C.c_void_p, C.c_int64]),
    ("fo_server_store_params_device", C.c_int, [C.c_void_p, C.c_void_p, C.c_int64]),
    ("fo_select_split", C.c_int, [C.c_void_p, C.c_void_p, C.c_int, C.c_void_p, C.c_void_p, C.c_int, C.c_void_p,
                                  C.POINTER(C.c_int), C.POINTER(C.c_double)]),
]


def lib():
    """Load libfedoptima.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise FedOptimaError(
                f"{LIB_PATH} is missing: build it with paper_2504_13850_gb300.build.build()")
        L = C.CDLL(LIB_PATH)
        for name, res, args in _SIGS:
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def exported_symbols():
    return [n for n, _, _ in _SIGS]


def last_error():
    return lib().fo_last_error().decode()


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        assert x.flags.c_contiguous
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        assert x.is_contiguous()
        return x.data_ptr()
    if isinstance(x, int):
        return x
    raise TypeError(type(x))


def _check(rc, what):
    if rc < 0:
        raise FedOptimaError(f"{what}: {STATUS.get(rc, rc)}: {last_error()}")
    return rc


def ops_to_c(ops):
    arr = (fo_op * len(ops))()
    for i, op in enumerate(ops):
        a = arr[i]
        a.kind = OP_KINDS[op["kind"]]
        a.in0 = op["in0"]
        a.in1 = op.get("in1", -1)
        a.cin = op.get("cin", op.get("c", 0))
        a.cout = op.get("cout", 0)
        a.k = op.get("k", 0)
        a.stride = op.get("stride", 1)
        a.bias = op.get("bias", 0)
        a.heads = op.get("heads", 0)
    return arr


class Server:
    """One FedOptima server (fo_server_*)."""

    def __init__(self, ops, K, omega, depth, batch, in_hwc, num_classes, dtype, lr, momentum,
                 seq=False, max_delay=2**31 - 1, policy=SCHED_COUNTER):
        L = lib()
        self._ops = ops_to_c(ops)
        self._opt = fo_optimizer(lr, momentum)
        self.cfg = fo_server_cfg(K, omega, depth, batch, in_hwc[0], in_hwc[1], in_hwc[2],
                                 num_classes, DTYPE_BF16 if dtype == "bf16" else DTYPE_F32,
                                 1 if seq else 0, max_delay, policy)
        h = C.c_void_p()
        _check(L.fo_server_create(self._ops, len(ops), C.byref(self._opt), C.byref(self.cfg),
                                  C.byref(h)), "fo_server_create")
        self.h = h
        self.K = K
        self.n_params = L.fo_server_num_params(h)

    @classmethod
    def from_config(cls, cfg, **over):
        kw = dict(ops=cfg["ops"], K=cfg["K"], omega=cfg["omega"], depth=cfg["depth"],
                  batch=cfg["batch"], in_hwc=cfg["in_hwc"], num_classes=cfg["classes"],
                  dtype=cfg["dtype"], lr=cfg["lr"], momentum=cfg["momentum"], seq=cfg["seq"])
        kw.update(over)
        return cls(**kw)

    def close(self):
        if getattr(self, "h", None):
            lib().fo_server_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # parameters -----------------------------------------------------------
    def set_params(self, theta):
        theta = np.ascontiguousarray(theta, np.float32)
        _check(lib().fo_server_set_params(self.h, _ptr(theta), theta.size), "set_params")

    def get_params(self):
        out = np.empty(self.n_params, np.float32)
        _check(lib().fo_server_get_params(self.h, _ptr(out), out.size), "get_params")
        return out

    def set_momentum(self, v):
        v = np.ascontiguousarray(v, np.float32)
        _check(lib().fo_server_set_momentum(self.h, _ptr(v), v.size), "set_momentum")

    def get_momentum(self):
        out = np.empty(self.n_params, np.float32)
        _check(lib().fo_server_get_momentum(self.h, _ptr(out), out.size), "get_momentum")
        return out

    # Algorithm 2 / 3 / 4 ----------------------------------------------------
    def enqueue_activations(self, device_id, acts, labels, lengths=None):
        """Returns (status, sender_on)."""
        on = C.c_int(-1)
        rc = lib().fo_enqueue_activations(self.h, device_id, _ptr(acts), _ptr(labels),
                                          _ptr(lengths), C.byref(on))
        if rc < 0 and rc != ERR_ARG:
            _check(rc, "enqueue_activations")
        return rc, on.value

    def server_step(self):
        """Returns (status, device_used, slot_used)."""
        k, slot = C.c_int(-1), C.c_int32(-1)
        rc = _check(lib().fo_server_step(self.h, C.byref(k), C.byref(slot)), "server_step")
        return rc, k.value, slot.value

    def read_losses(self, first, n):
        out = np.empty(n, np.float32)
        _check(lib().fo_read_losses(self.h, _ptr(out), first, n), "read_losses")
        return out

    def aggregate(self, global_, local, device_id, version):
        """Returns (status, new_version); global_ is a device buffer, local a
        device or host buffer (a host model is copied in by the library)."""
        nv = C.c_int32(-1)
        n = global_.numel() if hasattr(global_, "numel") else global_.size
        rc = lib().fo_aggregate(self.h, _ptr(global_), _ptr(local), n, device_id, version,
                                C.byref(nv))
        if rc < 0 and rc != ERR_ARG:
            _check(rc, "aggregate")
        return rc, nv.value

    # state ----------------------------------------------------------------
    def counters(self):
        out = np.zeros(self.K, np.uint64)
        _check(lib().fo_get_counters(self.h, _ptr(out)), "get_counters")
        return out

    def sender_status(self):
        out = np.zeros(self.K, np.uint8)
        _check(lib().fo_get_sender_status(self.h, _ptr(out)), "get_sender_status")
        return out

    def version(self):
        t, r = C.c_int32(), C.c_int32()
        _check(lib().fo_get_version(self.h, C.byref(t), C.byref(r)), "get_version")
        return t.value, r.value

    def set_device_active(self, k, active):
        return lib().fo_set_device_active(self.h, k, 1 if active else 0)

    def activation_bytes(self):
        return lib().fo_server_activation_bytes(self.h)

    def synchronize(self):
        _check(lib().fo_server_synchronize(self.h), "synchronize")

    def stream(self):
        return lib().fo_server_stream(self.h)

    def agg_stream(self):
        return lib().fo_server_agg_stream(self.h)

    def join_aggregations(self):
        _check(lib().fo_server_join_aggregations(self.h), "join_aggregations")

    def last_step_launches(self):
        return lib().fo_server_last_step_launches(self.h)

    def profile(self, enable):
        _check(lib().fo_server_profile(self.h, 1 if enable else 0), "profile")

    def kernel_times(self):
        """{name: (kernel launches, ms, algorithmic FLOPs, algorithmic bytes)}"""
        cap = 256
        names = (C.c_char_p * cap)()
        launches = (C.c_int64 * cap)()
        ms = (C.c_double * cap)()
        fl = (C.c_double * cap)()
        by = (C.c_double * cap)()
        n = C.c_int()
        _check(lib().fo_server_kernel_times(self.h, names, launches, ms, fl, by, cap, C.byref(n)),
               "kernel_times")
        return {names[i].decode(): (int(launches[i]), float(ms[i]), float(fl[i]), float(by[i]))
                for i in range(min(n.value, cap))}

    def profile_reset(self):
        _check(lib().fo_server_profile_reset(self.h), "profile_reset")

    def kernels_launched(self):
        return lib().fo_server_kernels_launched(self.h)

    def device_bytes(self):
        return lib().fo_server_device_bytes(self.h)

    def tensor(self, index):
        """(device pointer, (N, H, W, C), dtype) of the output of op index-1."""
        ptr, dims, dt = C.c_void_p(), (C.c_int64 * 4)(), C.c_int(0)
        _check(lib().fo_server_tensor(self.h, index, C.byref(ptr), dims, C.byref(dt)), "fo_server_tensor")
        return ptr.value, tuple(int(v) for v in dims), dt.value

    def params_device(self):
        """(device pointer, length) of the fp32 parameters in the padded layout."""
        ptr, n = C.c_void_p(), C.c_int64(0)
        _check(lib().fo_server_params_device(self.h, C.byref(ptr), C.byref(n)), "fo_server_params_device")
        return ptr.value, n.value

    def load_params_device(self, src_ptr, n):
        _check(lib().fo_server_load_params_device(self.h, C.c_void_p(src_ptr), n), "fo_server_load_params_device")

    def store_params_device(self, dst_ptr, n):
        _check(lib().fo_server_store_params_device(self.h, C.c_void_p(dst_ptr), n), "fo_server_store_params_device")

    def check_error(self):
        _check(lib().fo_server_error(self.h), "server_error")


class Scheduler:
    """Host-only Task Scheduler (fo_sched_*)."""

    def __init__(self, K, omega, depth, policy=SCHED_COUNTER):
        h = C.c_void_p()
        _check(lib().fo_sched_create(K, omega, depth, policy, C.byref(h)), "fo_sched_create")
        self.h, self.K = h, K

    def __del__(self):
        if getattr(self, "h", None):
            lib().fo_sched_destroy(self.h)
            self.h = None

    def put(self, k):
        slot, on = C.c_int32(-1), C.c_int(-1)
        rc = lib().fo_sched_put(self.h, k, C.byref(slot), C.byref(on))
        return rc, slot.value, on.value

    def get(self):
        k, slot = C.c_int(-1), C.c_int32(-1)
        rc = lib().fo_sched_get(self.h, C.byref(k), C.byref(slot))
        return rc, k.value, slot.value

    def set_active(self, k, active):
        return lib().fo_sched_set_active(self.h, k, 1 if active else 0)

    def counters(self):
        out = np.zeros(self.K, np.uint64)
        lib().fo_sched_counters(self.h, _ptr(out))
        return [int(v) for v in out]

    def sender_status(self):
        out = np.zeros(self.K, np.uint8)
        lib().fo_sched_sender_status(self.h, _ptr(out))
        return [int(v) for v in out]

    def queued(self, k=-1):
        return lib().fo_sched_queued(self.h, k)


def column_sums(x, out, stream=None):
    """out[c] = sum_r x[r][c] for a 2-D fp32 / bf16 device tensor x."""
    import torch
    dt = DTYPE_BF16 if x.dtype == torch.bfloat16 else DTYPE_F32
    return lib().fo_column_sums(_ptr(x), dt, x.shape[0], x.shape[1], _ptr(out), stream)


def column_sums_noalloc(x, out, stream=None):
    """column_sums with the partial sums in the library's fixed device array
    (no allocation); see fo_column_sums_noalloc for the size limit."""
    import torch
    dt = DTYPE_BF16 if x.dtype == torch.bfloat16 else DTYPE_F32
    return lib().fo_column_sums_noalloc(_ptr(x), dt, x.shape[0], x.shape[1], _ptr(out), stream)


def axpby_async(global_, local, alpha, stream=None):
    n = global_.numel() if hasattr(global_, "numel") else global_.size
    _check(lib().fo_axpby_async(_ptr(global_), _ptr(local), n, alpha, stream), "axpby_async")


def select_split(O, S, b, o, allowed=None):
    """Pre-processor split point (Eqs. 4-6) through fo_select_split: returns
    (status, l, cost) with l 1-based (split after layer l)."""
    O = np.ascontiguousarray(O, np.float64)
    S = np.ascontiguousarray(S, np.float64)
    b = np.ascontiguousarray(b, np.float64)
    o = np.ascontiguousarray(o, np.float64)
    al = None if allowed is None else np.ascontiguousarray(allowed, np.uint8)
    l, cost = C.c_int(0), C.c_double(0.0)
    rc = lib().fo_select_split(O.ctypes.data, S.ctypes.data, len(O), b.ctypes.data, o.ctypes.data, len(b),
                               None if al is None else al.ctypes.data, C.byref(l), C.byref(cost))
    return rc, l.value, cost.value
