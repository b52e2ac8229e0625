"""Thin ctypes binding of libadapm (include/adapm.h): argument marshalling only.

Every entry point of the C ABI has a method of the same name (without the
``adapm_`` prefix) on ParameterManager.  Arrays may be torch tensors on the
GPU or on the host (pinned or not) or numpy arrays; keys are passed as
32-bit integers, rows as float32.  All work runs in the library's CUDA
kernels; if the library is missing this module raises instead of falling
back to anything else.
"""
import ctypes
import os

import numpy as np

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libadapm.so")

OK, EINVAL, ERANGE, ENOMEM, ESTATE, ECUDA, ETIMEOUT = range(7)
STATUS_NAMES = {0: "OK", 1: "EINVAL", 2: "ERANGE", 3: "ENOMEM", 4: "ESTATE", 5: "ECUDA", 6: "ETIMEOUT"}
NUM_OPS = 8
OP_NAMES = ["intent", "advance", "pull", "push", "sync", "step", "push_kernel", "pull_kernel"]
NO_KEY = 0xFFFFFFFF
_CUDA_STREAM_LEGACY = 0x1

EXPORTS = [
    "adapm_create", "adapm_destroy", "adapm_intent", "adapm_advance_clock", "adapm_pull",
    "adapm_push", "adapm_sync", "adapm_wait", "adapm_mf_step", "adapm_complex_step",
    "adapm_sgns_step", "adapm_clock", "adapm_replica_keys", "adapm_replica_rows",
    "adapm_refcounts", "adapm_owners", "adapm_poisson_quantile", "adapm_read_main", "adapm_get_stats", "adapm_profile_enable",
    "adapm_profile_read", "adapm_kernel_launches", "adapm_push_noalloc", "adapm_last_error",
    "adapm_debug_fail_next_barrier", "adapm_debug_fail_next_launch",
]


class Config(ctypes.Structure):
    _fields_ = [
        ("num_keys", ctypes.c_uint64),
        ("value_len", ctypes.c_uint32),
        ("num_workers", ctypes.c_uint32),
        ("replica_capacity", ctypes.c_uint64),
        ("init_values", ctypes.c_void_p),
        ("stream", ctypes.c_void_p),
        ("relocate", ctypes.c_int32),
        ("action_timing", ctypes.c_int32),
        ("timing_alpha", ctypes.c_double),
        ("timing_p", ctypes.c_double),
        ("timing_lambda0", ctypes.c_double),
        ("delta_refresh", ctypes.c_int32),
        ("no_push_plans", ctypes.c_int32),
        ("pull_staging", ctypes.c_int32),
        ("no_early_events", ctypes.c_int32),
    ]


ACTION_TIMING = {"start": 0, "adaptive": 1, "signal": 2}


class Stats(ctypes.Structure):
    _fields_ = [
        ("live_replicas", ctypes.c_uint64),
        ("high_water", ctypes.c_uint64),
        ("capacity", ctypes.c_uint64),
        ("created", ctypes.c_uint64),
        ("destroyed", ctypes.c_uint64),
        ("last_push_unique", ctypes.c_uint64),
        ("push_rows", ctypes.c_uint64),
        ("push_unique", ctypes.c_uint64),
        ("sync_keys", ctypes.c_uint64),
        ("sync_replicas", ctypes.c_uint64),
        ("relocations", ctypes.c_uint64),
        ("sync_refreshed", ctypes.c_uint64),
        ("planned_pushes", ctypes.c_uint64),
        ("plan_misses", ctypes.c_uint64),
        ("early_advances", ctypes.c_uint64),
        ("early_undone", ctypes.c_uint64),
    ]


class AdaPMError(RuntimeError):
    def __init__(self, status, message):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


_lib = None


def load(path=LIB_PATH):
    """Load libadapm.so and declare its signatures (raises if it is missing)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build()")
    L = ctypes.CDLL(path)
    P, U32, U64, I64, F, I = (ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int64,
                              ctypes.c_float, ctypes.c_int)
    sig = {
        "adapm_create": [ctypes.POINTER(Config), ctypes.POINTER(P)],
        "adapm_destroy": [P],
        "adapm_intent": [P, U32, P, U64, I64, I64],
        "adapm_advance_clock": [P, U32],
        "adapm_pull": [P, U32, P, U64, P],
        "adapm_push": [P, U32, P, U64, P],
        "adapm_sync": [P],
        "adapm_wait": [P],
        "adapm_mf_step": [P, U32, P, P, P, U64, U32, I, F, F, P],
        "adapm_complex_step": [P, U32, P, P, P, P, U64, U32, U32, F, F, P],
        "adapm_sgns_step": [P, U32, P, P, P, U64, U32, U32, U32, U32, F, P],
        "adapm_clock": [P, U32, ctypes.POINTER(I64)],
        "adapm_replica_keys": [P, U32, P, U64, ctypes.POINTER(U64)],
        "adapm_replica_rows": [P, U32, P, U64, P, P, P],
        "adapm_refcounts": [P, U32, P, U64, P],
        "adapm_owners": [P, P, U64, P],
        "adapm_poisson_quantile": [ctypes.c_double, ctypes.c_double, ctypes.POINTER(I64)],
        "adapm_read_main": [P, P, U64, P],
        "adapm_get_stats": [P, ctypes.POINTER(Stats)],
        "adapm_profile_enable": [P, I],
        "adapm_profile_read": [P, P, P],
        "adapm_kernel_launches": [ctypes.POINTER(U64)],
        "adapm_push_noalloc": [P, U32, P, U64, P],
        "adapm_debug_fail_next_barrier": [P],
        "adapm_debug_fail_next_launch": [P],
    }
    for name, args in sig.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = ctypes.c_int
    L.adapm_last_error.argtypes = [P]
    L.adapm_last_error.restype = ctypes.c_char_p
    _lib = L
    return L


def kernel_launches():
    """Kernels launched by libadapm in this process so far."""
    v = ctypes.c_uint64()
    st = load().adapm_kernel_launches(ctypes.byref(v))
    if st != OK:
        raise AdaPMError(st, "adapm_kernel_launches")
    return v.value


def _torch():
    import torch
    return torch


class _Arr:
    """A pointer to a contiguous array and the object that keeps it alive."""

    __slots__ = ("ptr", "keep", "n")

    def __init__(self, ptr, keep, n):
        self.ptr, self.keep, self.n = ptr, keep, n


def _keys(a):
    if a is None:
        return _Arr(None, None, 0)
    if isinstance(a, np.ndarray) or isinstance(a, (list, tuple)):
        arr = np.ascontiguousarray(np.asarray(a, dtype=np.int64).astype(np.uint32))
        return _Arr(arr.ctypes.data if arr.size else None, arr, arr.size)
    torch = _torch()
    t = a.reshape(-1)
    if t.dtype != torch.int32:
        t = t.to(torch.int32)
    t = t.contiguous()
    return _Arr(t.data_ptr() if t.numel() else None, t, t.numel())


def _floats(a, dtype_np=np.float32):
    if a is None:
        return _Arr(None, None, 0)
    if isinstance(a, np.ndarray) or isinstance(a, (list, tuple)):
        arr = np.ascontiguousarray(np.asarray(a, dtype=dtype_np))
        return _Arr(arr.ctypes.data if arr.size else None, arr, arr.size)
    torch = _torch()
    t = a.contiguous()
    if t.dtype != torch.float32:
        t = t.to(torch.float32)
    return _Arr(t.data_ptr() if t.numel() else None, t, t.numel())


def _out_ptr(t):
    if isinstance(t, np.ndarray):
        assert t.flags["C_CONTIGUOUS"]
        return t.ctypes.data if t.size else None
    assert t.is_contiguous()
    return t.data_ptr() if t.numel() else None


def poisson_quantile(lam, p):
    """The p quantile of Poisson(lam) as the library's adaptive action timing computes it (host only)."""
    out = ctypes.c_int64()
    st = load().adapm_poisson_quantile(float(lam), float(p), ctypes.byref(out))
    if st != OK:
        raise AdaPMError(st, "adapm_poisson_quantile: need lam > 0 and 0 < p < 1")
    return out.value


class ParameterManager:
    """One adapm context (adapm_create).  Device arrays are used in place; host arrays are copied.

    relocate        move a key to its only worker with active intent instead of replicating it (Sec. 4.1)
    action_timing   "start" (act when an intent becomes active), "adaptive" (Algorithm 1 at each sync, with
                    timing_alpha / timing_p / timing_lambda0, 0 = the paper's 0.1 / 0.9999 / 10) or "signal"
    delta_refresh   versioned refresh: sync leaves a sole holder's value when nobody else wrote the key
    push_plans      sort each intent's keys beside the library stream and let a push with the same keys
                    use that sort (adapm_intent); False sorts every push itself
    pull_staging    pull rows through shared memory with bulk copies instead of through registers
    early_events    compute the refcount changes of a worker's next advance beside its pull and push
                    (adapm_advance_clock); False computes them in the advance
    """

    def __init__(self, num_keys, value_len, num_workers, replica_capacity=0, init_values=None,
                 stream=None, relocate=False, action_timing="start", timing_alpha=0.0, timing_p=0.0,
                 timing_lambda0=0.0, delta_refresh=False, push_plans=True, pull_staging=False,
                 early_events=True):
        self._lib = load()
        torch = _torch()
        if stream is None:
            stream = torch.cuda.current_stream()
        self.stream = stream
        self.K, self.D, self.W = int(num_keys), int(value_len), int(num_workers)
        init = _floats(init_values)
        if init.ptr is not None and init.n != self.K * self.D:
            raise ValueError("init_values must hold num_keys * value_len floats")
        # torch's default stream has handle 0; the ABI reads NULL as "make a
        # stream of your own", so name the legacy default stream (0x1) instead
        handle = stream.cuda_stream or _CUDA_STREAM_LEGACY
        self.relocate = bool(relocate)
        if action_timing not in ACTION_TIMING:
            raise ValueError(f"action_timing must be one of {sorted(ACTION_TIMING)}")
        self.action_timing = action_timing
        cfg = Config(self.K, self.D, self.W, int(replica_capacity), init.ptr,
                     ctypes.c_void_p(handle), int(self.relocate), ACTION_TIMING[action_timing],
                     float(timing_alpha), float(timing_p), float(timing_lambda0), int(bool(delta_refresh)),
                     int(not push_plans), int(bool(pull_staging)), int(not early_events))
        h = ctypes.c_void_p()
        st = self._lib.adapm_create(ctypes.byref(cfg), ctypes.byref(h))
        if st != OK:
            raise AdaPMError(st, "adapm_create failed")
        self._h = h

    # -- plumbing ------------------------------------------------------------
    def _check(self, st):
        if st != OK:
            msg = self._lib.adapm_last_error(self._h)
            raise AdaPMError(st, msg.decode() if msg else "")

    def close(self):
        if getattr(self, "_h", None):
            self._lib.adapm_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _new_rows(self, n, like):
        torch = _torch()
        if isinstance(like, np.ndarray):
            return np.empty((n, self.D), dtype=np.float32)
        dev = like.device if like is not None and hasattr(like, "device") else torch.device("cuda")
        pin = dev.type == "cpu"
        return torch.empty((n, self.D), dtype=torch.float32, device=dev, pin_memory=pin)

    # -- the ABI -------------------------------------------------------------
    def intent(self, worker, keys, clock_start, clock_end):
        k = _keys(keys)
        self._check(self._lib.adapm_intent(self._h, worker, k.ptr, k.n, int(clock_start), int(clock_end)))

    def advance_clock(self, worker):
        self._check(self._lib.adapm_advance_clock(self._h, worker))

    def pull(self, worker, keys, out=None):
        k = _keys(keys)
        if out is None:
            out = self._new_rows(k.n, keys)
        self._check(self._lib.adapm_pull(self._h, worker, k.ptr, k.n, _out_ptr(out)))
        return out

    def push(self, worker, keys, deltas):
        k = _keys(keys)
        d = _floats(deltas)
        if d.n != k.n * self.D:
            raise ValueError("deltas must hold len(keys) * value_len floats")
        self._check(self._lib.adapm_push(self._h, worker, k.ptr, k.n, d.ptr))

    def push_noalloc(self, worker, keys, deltas):
        """adapm_push_noalloc: device tensors only; no allocation by the library."""
        k = _keys(keys)
        d = _floats(deltas)
        if d.n != k.n * self.D:
            raise ValueError("deltas must hold len(keys) * value_len floats")
        self._check(self._lib.adapm_push_noalloc(self._h, worker, k.ptr, k.n, d.ptr))

    def last_error(self):
        """adapm_last_error: the message of the last error returned on this context ("" if none)."""
        msg = self._lib.adapm_last_error(self._h)
        return msg.decode() if msg else ""

    def debug_fail_next_barrier(self):
        """Test hook: the next push's sort gives up its grid-barrier wait (ADAPM_ETIMEOUT at wait)."""
        self._check(self._lib.adapm_debug_fail_next_barrier(self._h))

    def debug_fail_next_launch(self):
        """Test hook: the next call that launches kernels returns ADAPM_ECUDA as after a launch failure."""
        self._check(self._lib.adapm_debug_fail_next_launch(self._h))

    def sync(self):
        self._check(self._lib.adapm_sync(self._h))

    def wait(self):
        self._check(self._lib.adapm_wait(self._h))

    def _loss_buf(self, loss_out):
        if loss_out is not None:
            return loss_out, _out_ptr(loss_out)
        return None, None

    def mf_step(self, worker, row_keys, col_keys, vals, dim, adagrad, lr, eps=1e-8, loss_out=None):
        r, c, v = _keys(row_keys), _keys(col_keys), _floats(vals)
        lo, lp = self._loss_buf(loss_out)
        self._check(self._lib.adapm_mf_step(self._h, worker, r.ptr, c.ptr, v.ptr, r.n, dim,
                                            int(bool(adagrad)), lr, eps, lp))
        return lo

    def complex_step(self, worker, heads, rels, tails, neg_tails, n_neg, dim, lr, eps=1e-8,
                     loss_out=None):
        h, r, t, ng = _keys(heads), _keys(rels), _keys(tails), _keys(neg_tails)
        lo, lp = self._loss_buf(loss_out)
        self._check(self._lib.adapm_complex_step(self._h, worker, h.ptr, r.ptr, t.ptr, ng.ptr, h.n,
                                                 n_neg, dim, lr, eps, lp))
        return lo

    def sgns_step(self, worker, centres, contexts, negatives, n_ctx, n_neg, vocab, dim, lr,
                  loss_out=None):
        c, x, ng = _keys(centres), _keys(contexts), _keys(negatives)
        lo, lp = self._loss_buf(loss_out)
        self._check(self._lib.adapm_sgns_step(self._h, worker, c.ptr, x.ptr, ng.ptr, c.n, n_ctx,
                                              n_neg, vocab, dim, lr, lp))
        return lo

    # -- inspection ------------------------------------------------------------
    def clock(self, worker):
        v = ctypes.c_int64()
        self._check(self._lib.adapm_clock(self._h, worker, ctypes.byref(v)))
        return v.value

    def replica_keys(self, worker):
        n = ctypes.c_uint64()
        self._check(self._lib.adapm_replica_keys(self._h, worker, None, 0, ctypes.byref(n)))
        out = np.empty(n.value, dtype=np.uint32)
        if n.value:
            self._check(self._lib.adapm_replica_keys(self._h, worker, out.ctypes.data, n.value,
                                                     ctypes.byref(n)))
        return out.astype(np.int64)

    def replica_rows(self, worker, keys):
        k = _keys(keys)
        val = np.zeros((k.n, self.D), np.float32)
        acc = np.zeros((k.n, self.D), np.float32)
        has = np.zeros(k.n, np.uint8)
        self._check(self._lib.adapm_replica_rows(self._h, worker, k.ptr, k.n, _out_ptr(val),
                                                 _out_ptr(acc), _out_ptr(has)))
        return val, acc, has.astype(bool)

    def refcounts(self, worker, keys):
        k = _keys(keys)
        out = np.zeros(k.n, np.uint32)
        self._check(self._lib.adapm_refcounts(self._h, worker, k.ptr, k.n, _out_ptr(out)))
        return out.astype(np.int64)

    def owners(self, keys):
        """Owner worker of each key, -1 while it is at its home."""
        k = _keys(keys)
        out = np.zeros(k.n, np.int32)
        self._check(self._lib.adapm_owners(self._h, k.ptr, k.n, _out_ptr(out)))
        return out

    def read_main(self, keys):
        k = _keys(keys)
        out = np.zeros((k.n, self.D), np.float32)
        self._check(self._lib.adapm_read_main(self._h, k.ptr, k.n, _out_ptr(out)))
        return out

    def stats(self):
        s = Stats()
        self._check(self._lib.adapm_get_stats(self._h, ctypes.byref(s)))
        return {f: getattr(s, f) for f, _ in Stats._fields_}

    def profile_enable(self, enable=True):
        self._check(self._lib.adapm_profile_enable(self._h, int(bool(enable))))

    def profile_read(self):
        ms = (ctypes.c_double * NUM_OPS)()
        calls = (ctypes.c_uint64 * NUM_OPS)()
        self._check(self._lib.adapm_profile_read(self._h, ms, calls))
        return {OP_NAMES[i]: (ms[i], calls[i]) for i in range(NUM_OPS)}
