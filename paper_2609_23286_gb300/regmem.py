"""Thin ctypes binding of libregmem.so (include/regmem.h).

The functions carry the C names and only marshal arguments: handles are
integers, tensors may be passed as torch tensors (their data_ptr() is used)
or as raw integer addresses.  Every compute step runs inside the library.
A negative status raises RegmemError with the library's message.  Loading
fails loudly when the library has not been built: there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libregmem.so")
# the same library with the kernels' range guards compiled in (build(checks=True))
CHECKED_LIB_PATH = os.path.join(_HERE, "libregmem_checked.so")

OK, ERR_ARG, ERR_STATE, ERR_CAPACITY, ERR_CUDA, ERR_UNSUPPORTED, ERR_TIMEOUT = 0, -1, -2, -3, -4, -5, -6
ERR_DEVICE_CHECK = -7

# Every exported entry point of include/regmem.h with its ctypes signature.
_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_SIGNATURES = {
    "regmem_create": (ctypes.c_int, [ctypes.POINTER(_P), _I32, _I32, _I32, _I32]),
    "regmem_set_frame": (ctypes.c_int, [_P, _P]),
    "regmem_set_stream": (ctypes.c_int, [_P, _P]),
    "regmem_set_overlap": (ctypes.c_int, [_P, _I32]),
    "regmem_join": (ctypes.c_int, [_P]),
    "regmem_attend_frame": (ctypes.c_int, [_P, _I32, _P, _P, _P, _P, _P]),
    "regmem_attend_frame_host": (ctypes.c_int, [_P, _I32, _P, _P, _P, _P, _P]),
    "regmem_admit": (ctypes.c_int, [_P, _I32, _I32, _P]),
    "regmem_admit_shared": (ctypes.c_int, [_P, _I32, _I32, _P]),
    "regmem_attend_admit": (ctypes.c_int, [_P, _I32, _P, _P, _P, _P, _P, _I32, _P]),
    "regmem_attend_admit_shared": (ctypes.c_int, [_P, _I32, _P, _P, _P, _P, _P, _I32, _P]),
    "regmem_attend_admit_host": (ctypes.c_int, [_P, _I32, _P, _P, _P, _P, _P, _I32]),
    "regmem_frame_attention": (ctypes.c_int, [_P, _P, _P, _P, _P]),
    "regmem_reset": (ctypes.c_int, [_P]),
    "regmem_memory_len": (ctypes.c_int, [_P, _I32, ctypes.POINTER(ctypes.c_int64)]),
    "regmem_capacity": (ctypes.c_int, [_P, ctypes.POINTER(ctypes.c_int64)]),
    "regmem_export_bank": (ctypes.c_int, [_P, _I32, _P, _P]),
    "regmem_import_bank": (ctypes.c_int, [_P, _I32, _P, _P, ctypes.c_int64]),
    "regmem_copy_lse": (ctypes.c_int, [_P, _P]),
    "regmem_synchronize": (ctypes.c_int, [_P]),
    "regmem_attend_frame_noalloc": (ctypes.c_int, [_P, _I32, _P, _P, _P, _P, _P, ctypes.c_int64,
                                                   ctypes.c_int64, _P, _P, _P, _P]),
    "regmem_debug_set": (ctypes.c_int, [_P, ctypes.c_int64, _I32]),
    "regmem_profile_enable": (ctypes.c_int, [_P, _I32]),
    "regmem_profile_read": (ctypes.c_int, [_P, _P]),
    "regmem_last_error": (ctypes.c_char_p, [_P]),
    "regmem_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "regmem_destroy": (None, [_P]),
}


class FrameDesc(ctypes.Structure):
    """regmem_frame_desc."""
    _fields_ = [("n_tokens", _I32), ("n_special", _I32), ("grid_h", _I32), ("grid_w", _I32),
                ("ds", _I32), ("max_frames", _I32), ("scale", ctypes.c_float),
                ("candidates", _I32)]


class Profile(ctypes.Structure):
    """regmem_profile."""
    _fields_ = [("launches_attention", ctypes.c_int64),
                ("launches_saliency", ctypes.c_int64), ("launches_admit", ctypes.c_int64),
                ("launches_anchor", ctypes.c_int64), ("launches_combine", ctypes.c_int64),
                ("attention_timed", ctypes.c_int64),
                ("attention_ms", ctypes.c_double), ("attention_flops", ctypes.c_double),
                ("attention_bytes", ctypes.c_double), ("attention_ctas", ctypes.c_int32),
                ("attention_ctas_per_sm", ctypes.c_int32), ("merge_ms", ctypes.c_double),
                ("attention_clocked", ctypes.c_int64), ("attention_clock_ms", ctypes.c_double),
                ("attention_clock_flops", ctypes.c_double),
                ("launches_frame_attention", ctypes.c_int64),
                ("frame_attention_clocked", ctypes.c_int64),
                ("frame_attention_clock_ms", ctypes.c_double),
                ("frame_attention_clock_flops", ctypes.c_double)]

    def as_dict(self):
        return {f: getattr(self, f) for f, _ in self._fields_}

    def launches(self):
        return (self.launches_attention + self.launches_saliency + self.launches_admit
                + self.launches_anchor + self.launches_combine)


class RegmemError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{status_string(status)}: {msg}")
        self.status = status


_lib = None


def load(path: str | None = None):
    """Load libregmem.so (once).  Raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"{p} is missing: build it with __graft_entry__.build() "
                           "(python -m paper_2609_23286_gb300.build)")
    lib = ctypes.CDLL(p)
    for name, (res, args) in _SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):          # numpy array
        return x.ctypes.data
    raise TypeError(f"cannot take the address of {type(x)}")


def _check(h, st: int):
    if st < 0:
        msg = load().regmem_last_error(h)
        raise RegmemError(st, msg.decode() if msg else "")
    return st


def status_string(st: int) -> str:
    return load().regmem_status_string(st).decode()


def regmem_create(layers: int, heads: int, head_dim: int, budget: int) -> int:
    h = _P()
    st = load().regmem_create(ctypes.byref(h), layers, heads, head_dim, budget)
    if st < 0:
        raise RegmemError(st, "regmem_create rejected its arguments")
    return h.value


def regmem_set_frame(h, n_tokens, n_special, grid_h, grid_w, ds=2, max_frames=1, scale=0.0,
                     candidates=0):
    fd = FrameDesc(n_tokens, n_special, grid_h, grid_w, ds, max_frames, scale, candidates)
    return _check(h, load().regmem_set_frame(h, ctypes.byref(fd)))


def regmem_set_stream(h, stream):
    return _check(h, load().regmem_set_stream(h, _stream_ptr(stream)))


def regmem_set_overlap(h, on):
    return _check(h, load().regmem_set_overlap(h, int(on)))


def regmem_join(h):
    return _check(h, load().regmem_join(h))


def _stream_ptr(stream):
    if stream is None or isinstance(stream, int):
        return stream
    return stream.cuda_stream  # torch.cuda.Stream


def regmem_attend_frame(h, layer, Q, K, V, out, saliency):
    return _check(h, load().regmem_attend_frame(h, layer, _ptr(Q), _ptr(K), _ptr(V), _ptr(out),
                                                _ptr(saliency)))


def regmem_attend_frame_host(h, layer, Q, K, V, out, saliency):
    return _check(h, load().regmem_attend_frame_host(h, layer, _ptr(Q), _ptr(K), _ptr(V),
                                                     _ptr(out), _ptr(saliency)))


def regmem_admit(h, layer, k, idx_out=None):
    return _check(h, load().regmem_admit(h, layer, k, _ptr(idx_out)))


def regmem_admit_shared(h, layer, k, idx_out=None):
    return _check(h, load().regmem_admit_shared(h, layer, k, _ptr(idx_out)))


def regmem_attend_admit(h, layer, Q, K, V, out, saliency, k, idx_out=None):
    return _check(h, load().regmem_attend_admit(h, layer, _ptr(Q), _ptr(K), _ptr(V), _ptr(out),
                                                _ptr(saliency), k, _ptr(idx_out)))


def regmem_attend_admit_shared(h, layer, Q, K, V, out, saliency, k, idx_out=None):
    return _check(h, load().regmem_attend_admit_shared(h, layer, _ptr(Q), _ptr(K), _ptr(V), _ptr(out),
                                                       _ptr(saliency), k, _ptr(idx_out)))


def regmem_attend_admit_host(h, layer, Q, K, V, out, saliency, k):
    return _check(h, load().regmem_attend_admit_host(h, layer, _ptr(Q), _ptr(K), _ptr(V),
                                                     _ptr(out), _ptr(saliency), k))


def regmem_frame_attention(h, Q, K, V, out):
    return _check(h, load().regmem_frame_attention(h, _ptr(Q), _ptr(K), _ptr(V), _ptr(out)))


def regmem_reset(h):
    return _check(h, load().regmem_reset(h))


def regmem_memory_len(h, layer) -> int:
    v = ctypes.c_int64()
    _check(h, load().regmem_memory_len(h, layer, ctypes.byref(v)))
    return v.value


def regmem_capacity(h) -> int:
    v = ctypes.c_int64()
    _check(h, load().regmem_capacity(h, ctypes.byref(v)))
    return v.value


def regmem_export_bank(h, layer, hostK, hostV):
    return _check(h, load().regmem_export_bank(h, layer, _ptr(hostK), _ptr(hostV)))


def regmem_import_bank(h, layer, hostK, hostV, length):
    return _check(h, load().regmem_import_bank(h, layer, _ptr(hostK), _ptr(hostV), length))


def regmem_copy_lse(h, dst):
    return _check(h, load().regmem_copy_lse(h, _ptr(dst)))


def regmem_synchronize(h):
    return _check(h, load().regmem_synchronize(h))


def regmem_attend_frame_noalloc(n_special, grid_h, grid_w, heads, Q, K, V, bankK, bankV,
                                bank_rows, M, out, saliency, status=None, stream=None, ds=2,
                                scale=0.0):
    """Handle-free attend step whose scratch is a fixed device array inside
    the library (no device allocation).  `status` (a device int32, zeroed by
    the caller) is required: the kernels record an expired wait there."""
    fd = FrameDesc(n_special + grid_h * grid_w, n_special, grid_h, grid_w, ds, 1, scale, 0)
    st = load().regmem_attend_frame_noalloc(ctypes.byref(fd), heads, _ptr(Q), _ptr(K), _ptr(V),
                                            _ptr(bankK), _ptr(bankV), bank_rows, M, _ptr(out),
                                            _ptr(saliency), _ptr(status), _stream_ptr(stream))
    if st < 0:
        raise RegmemError(st, "regmem_attend_frame_noalloc rejected the call")
    return st


def regmem_debug_set(h, wait_limit_us=2000000, skip_kv_load=-1):
    """Failure-detection hook: bounded-wait limit of the attention kernel and
    a one-shot skipped K/V load in its next launch."""
    return _check(h, load().regmem_debug_set(h, int(wait_limit_us), int(skip_kv_load)))


def regmem_profile_enable(h, time_attention=1):
    return _check(h, load().regmem_profile_enable(h, int(time_attention)))


def regmem_profile_read(h) -> Profile:
    p = Profile()
    _check(h, load().regmem_profile_read(h, ctypes.byref(p)))
    return p


def regmem_last_error(h) -> str:
    return load().regmem_last_error(h).decode()


def regmem_status_string(st: int) -> str:
    return status_string(st)


def regmem_destroy(h):
    load().regmem_destroy(h)


class RegMem:
    """Owning wrapper around a handle (context manager)."""

    def __init__(self, layers, heads, head_dim, budget):
        self.h = regmem_create(layers, heads, head_dim, budget)
        self.layers, self.heads, self.head_dim, self.budget = layers, heads, head_dim, budget

    def set_frame(self, n_special, grid_h, grid_w, ds=2, max_frames=1, scale=0.0, candidates=0):
        self.N = n_special + grid_h * grid_w
        return regmem_set_frame(self.h, self.N, n_special, grid_h, grid_w, ds, max_frames,
                                scale, candidates)

    def set_stream(self, stream):
        return regmem_set_stream(self.h, stream)

    def set_overlap(self, on):
        return regmem_set_overlap(self.h, on)

    def join(self):
        return regmem_join(self.h)

    def attend_frame(self, layer, Q, K, V, out, saliency):
        return regmem_attend_frame(self.h, layer, Q, K, V, out, saliency)

    def attend_frame_host(self, layer, Q, K, V, out, saliency):
        return regmem_attend_frame_host(self.h, layer, Q, K, V, out, saliency)

    def admit(self, layer, k, idx_out=None):
        return regmem_admit(self.h, layer, k, idx_out)

    def admit_shared(self, layer, k, idx_out=None):
        """One index set for all heads (no head-specific retention)."""
        return regmem_admit_shared(self.h, layer, k, idx_out)

    def attend_admit(self, layer, Q, K, V, out, saliency, k, idx_out=None):
        return regmem_attend_admit(self.h, layer, Q, K, V, out, saliency, k, idx_out)

    def attend_admit_shared(self, layer, Q, K, V, out, saliency, k, idx_out=None):
        """attend_frame + admit_shared in one call (side stream with overlap)."""
        return regmem_attend_admit_shared(self.h, layer, Q, K, V, out, saliency, k, idx_out)

    def attend_admit_host(self, layer, Q, K, V, out, saliency, k):
        return regmem_attend_admit_host(self.h, layer, Q, K, V, out, saliency, k)

    def frame_attention(self, Q, K, V, out):
        return regmem_frame_attention(self.h, Q, K, V, out)

    def reset(self):
        return regmem_reset(self.h)

    def memory_len(self, layer):
        return regmem_memory_len(self.h, layer)

    def capacity(self):
        return regmem_capacity(self.h)

    def export_bank(self, layer, hostK, hostV):
        return regmem_export_bank(self.h, layer, hostK, hostV)

    def import_bank(self, layer, hostK, hostV, length):
        return regmem_import_bank(self.h, layer, hostK, hostV, length)

    def copy_lse(self, dst):
        return regmem_copy_lse(self.h, dst)

    def synchronize(self):
        return regmem_synchronize(self.h)

    def debug_set(self, wait_limit_us=2000000, skip_kv_load=-1):
        return regmem_debug_set(self.h, wait_limit_us, skip_kv_load)

    def profile_enable(self, time_attention=1):
        return regmem_profile_enable(self.h, time_attention)

    def profile_read(self) -> Profile:
        return regmem_profile_read(self.h)

    def close(self):
        if self.h:
            regmem_destroy(self.h)
            self.h = 0

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
