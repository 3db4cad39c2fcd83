"""Python binding of the C ABI in include/lora.h (argument marshalling only).

Every function has the name and argument order of its C counterpart.  Device
buffers may be passed as integers (device addresses) or as CUDA tensors of
any object with `data_ptr()`; `stream` may be an integer cudaStream_t, an
object with a `cuda_stream` attribute (a torch.cuda.Stream), or None for
the caller's current torch stream.  A non-zero return code raises LoraError.
The compute runs only in the CUDA library: if it is not built, loading
fails with an error; there is no other code path.
"""
from __future__ import annotations

import ctypes
import os

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "liblora_gb300.so")
_lib = None

LORA_OK = 0
LORA_EINVAL = -1
LORA_ENULL = -2
LORA_EALIGN = -3
LORA_ECUDA = -4
LORA_ETIMEOUT = -5
LORA_EWORKSPACE = -6
LORA_EDEVICE = -7
LORA_ESCRATCH = -8

LORA_FWD = 1
LORA_BWD = 2
LORA_FWD_BWD = 3

# every symbol that include/lora.h declares
EXPORTS = ("lora_workspace_size", "lora_linear_fwd", "lora_linear_fwd_noalloc", "lora_linear_bwd",
           "lora_linear_fwd_q4", "lora_linear_bwd_q4", "lora_stack_workspace_size",
           "lora_stack_step", "lora_stack_ckpt_workspace_size", "lora_stack_ckpt", "lora_ce_workspace_size",
           "lora_ce_fwd_bwd", "lora_topk_workspace_size", "lora_topk_table", "lora_wait_selftest",
           "lora_read_status", "lora_set_wait_limit_ns", "lora_launch_count",
           "lora_profile_begin", "lora_profile_begin_kinds", "lora_profile_end", "lora_strerror", "lora_version",
           "lora_last_error")

LORA_KERNEL_GEMM_FWD = 0
LORA_KERNEL_GEMM_BWD = 1
LORA_KERNEL_ROWPROJ = 2
LORA_KERNEL_COLPROJ = 3
LORA_KERNEL_PAD = 4
LORA_KERNEL_KINDS = 5
KERNEL_NAMES = ("gemm_fwd", "gemm_bwd", "rowproj", "colproj", "pad")


class LoraError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        msg = library().lora_strerror(code).decode() if _lib is not None else str(code)
        super().__init__(f"{where}: {msg} ({code})")


class lora_shape(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int64), ("d_in", ctypes.c_int64), ("d_out", ctypes.c_int64),
                ("rank", ctypes.c_int64), ("scale", ctypes.c_float)]


class lora_q4_weight(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("params", ctypes.c_void_p)]


class lora_proj(ctypes.Structure):
    _fields_ = [("shape", lora_shape),
                ("x", ctypes.c_void_p), ("W", ctypes.c_void_p), ("A", ctypes.c_void_p), ("B", ctypes.c_void_p),
                ("dy", ctypes.c_void_p), ("y", ctypes.c_void_p), ("su", ctypes.c_void_p), ("dx", ctypes.c_void_p),
                ("dA", ctypes.c_void_p), ("dB", ctypes.c_void_p), ("Wq", lora_q4_weight)]


class lora_ce_args(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int64), ("d", ctypes.c_int64), ("V", ctypes.c_int64),
                ("h", ctypes.c_void_p), ("E", ctypes.c_void_p), ("targets", ctypes.c_void_p),
                ("mask", ctypes.c_void_p), ("topk", ctypes.c_void_p), ("ld_topk", ctypes.c_int64),
                ("k", ctypes.c_int64), ("loss", ctypes.c_void_p), ("token_loss", ctypes.c_void_p),
                ("dh", ctypes.c_void_p), ("vocab", ctypes.c_void_p), ("counts", ctypes.c_void_p)]


def library(path: str = _LIB_PATH) -> ctypes.CDLL:
    """Load the CUDA library (once).  Raises OSError if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise OSError(f"CUDA library not built: {path} (run paper_2606_19528_gb300.build)")
        lib = ctypes.CDLL(path)
        vp, sz, i32, i64 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_int64
        P = ctypes.POINTER
        lib.lora_workspace_size.argtypes = [P(lora_shape), i32, P(sz)]
        lib.lora_linear_fwd.argtypes = [P(lora_shape), vp, vp, vp, vp, vp, vp, vp, sz, vp]
        lib.lora_linear_fwd_noalloc.argtypes = [P(lora_shape), vp, vp, vp, vp, vp, vp, vp]
        lib.lora_linear_bwd.argtypes = [P(lora_shape), vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
        lib.lora_linear_fwd_q4.argtypes = [P(lora_shape), vp, P(lora_q4_weight), vp, vp, vp, vp, vp, sz, vp]
        lib.lora_linear_bwd_q4.argtypes = [P(lora_shape), vp, vp, P(lora_q4_weight), vp, vp, vp, vp, vp, vp, vp, sz,
                                           vp]
        lib.lora_stack_workspace_size.argtypes = [P(lora_proj), i32, i32, P(sz)]
        lib.lora_stack_step.argtypes = [P(lora_proj), i32, i32, vp, sz, vp]
        lib.lora_stack_ckpt_workspace_size.argtypes = [P(lora_proj), i32, i32, P(sz)]
        lib.lora_stack_ckpt.argtypes = [P(lora_proj), i32, i32, vp, sz, vp]
        lib.lora_ce_workspace_size.argtypes = [P(lora_ce_args), P(sz)]
        lib.lora_ce_fwd_bwd.argtypes = [P(lora_ce_args), vp, sz, vp]
        lib.lora_topk_workspace_size.argtypes = [i64, i64, i64, P(sz)]
        lib.lora_topk_table.argtypes = [vp, i64, i64, i64, vp, vp, sz, vp]
        lib.lora_wait_selftest.argtypes = [i64, vp]
        lib.lora_read_status.argtypes = [vp, P(i32), i32]
        lib.lora_set_wait_limit_ns.argtypes = [i64]
        lib.lora_launch_count.argtypes = []
        lib.lora_profile_begin.argtypes = []
        lib.lora_profile_begin_kinds.argtypes = [ctypes.c_uint32]
        lib.lora_profile_end.argtypes = [P(ctypes.c_double), P(i64)]
        lib.lora_strerror.argtypes = [i32]
        lib.lora_strerror.restype = ctypes.c_char_p
        lib.lora_version.argtypes = []
        lib.lora_last_error.argtypes = []
        for name in EXPORTS:
            if name != "lora_strerror":
                getattr(lib, name).restype = i32
        lib.lora_launch_count.restype = i64
        _lib = lib
    return _lib


def _ptr(a):
    if a is None:
        return None
    if isinstance(a, int):
        return a
    return a.data_ptr()


def _stream(s):
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(rc: int, where: str):
    if rc != LORA_OK:
        raise LoraError(rc, where)


def make_shape(T, d_in, d_out, rank, scale) -> lora_shape:
    return lora_shape(int(T), int(d_in), int(d_out), int(rank), float(scale))


def make_q4(codes, params) -> lora_q4_weight:
    """4-bit base weight: codes [d_out, d_in / 2] bytes and (s, b) pairs
    [d_out, d_in / 64, 2] bf16 (layout in include/lora.h)."""
    return lora_q4_weight(_ptr(codes), _ptr(params))


def make_proj(shape: lora_shape, x=None, W=None, A=None, B=None, dy=None, y=None, su=None, dx=None, dA=None,
              dB=None, Wq=None) -> lora_proj:
    return lora_proj(shape, _ptr(x), _ptr(W), _ptr(A), _ptr(B), _ptr(dy), _ptr(y), _ptr(su), _ptr(dx), _ptr(dA),
                     _ptr(dB), Wq if Wq is not None else lora_q4_weight(None, None))


def lora_workspace_size(shape: lora_shape, mode: int) -> int:
    n = ctypes.c_size_t(0)
    _check(library().lora_workspace_size(ctypes.byref(shape), mode, ctypes.byref(n)), "lora_workspace_size")
    return n.value


def lora_linear_fwd(shape, x, W, A, B, y, su, workspace, workspace_bytes, stream=None) -> None:
    _check(library().lora_linear_fwd(ctypes.byref(shape), _ptr(x), _ptr(W), _ptr(A), _ptr(B), _ptr(y), _ptr(su),
                                     _ptr(workspace), int(workspace_bytes), _stream(stream)), "lora_linear_fwd")


def lora_linear_fwd_noalloc(shape, x, W, A, B, y, su, stream=None) -> None:
    """Forward without a workspace argument (scratch in a fixed 4 MiB array
    inside the library), for callers that cannot allocate device memory when
    they call; see include/lora.h."""
    _check(library().lora_linear_fwd_noalloc(ctypes.byref(shape), _ptr(x), _ptr(W), _ptr(A), _ptr(B), _ptr(y),
                                             _ptr(su), _stream(stream)), "lora_linear_fwd_noalloc")


def lora_linear_bwd(shape, dy, x, W, A, B, su, dx, dA, dB, workspace, workspace_bytes, stream=None) -> None:
    _check(library().lora_linear_bwd(ctypes.byref(shape), _ptr(dy), _ptr(x), _ptr(W), _ptr(A), _ptr(B), _ptr(su),
                                     _ptr(dx), _ptr(dA), _ptr(dB), _ptr(workspace), int(workspace_bytes),
                                     _stream(stream)), "lora_linear_bwd")


def lora_linear_fwd_q4(shape, x, Wq: lora_q4_weight, A, B, y, su, workspace, workspace_bytes, stream=None) -> None:
    _check(library().lora_linear_fwd_q4(ctypes.byref(shape), _ptr(x), ctypes.byref(Wq), _ptr(A), _ptr(B), _ptr(y),
                                        _ptr(su), _ptr(workspace), int(workspace_bytes), _stream(stream)),
           "lora_linear_fwd_q4")


def lora_linear_bwd_q4(shape, dy, x, Wq: lora_q4_weight, A, B, su, dx, dA, dB, workspace, workspace_bytes,
                       stream=None) -> None:
    _check(library().lora_linear_bwd_q4(ctypes.byref(shape), _ptr(dy), _ptr(x), ctypes.byref(Wq), _ptr(A), _ptr(B),
                                        _ptr(su), _ptr(dx), _ptr(dA), _ptr(dB), _ptr(workspace),
                                        int(workspace_bytes), _stream(stream)), "lora_linear_bwd_q4")


def _proj_array(projs):
    arr = (lora_proj * len(projs))(*projs)
    return arr


def lora_stack_workspace_size(projs, mode: int) -> int:
    arr = _proj_array(projs)
    n = ctypes.c_size_t(0)
    _check(library().lora_stack_workspace_size(arr, len(projs), mode, ctypes.byref(n)), "lora_stack_workspace_size")
    return n.value


def lora_stack_step(projs, mode: int, workspace, workspace_bytes, stream=None) -> None:
    arr = _proj_array(projs)
    _check(library().lora_stack_step(arr, len(projs), mode, _ptr(workspace), int(workspace_bytes),
                                     _stream(stream)), "lora_stack_step")


def lora_stack_ckpt_workspace_size(layers) -> int:
    """`layers`: a list of layers, each a list of projections (same count)."""
    n_per = len(layers[0])
    arr = _proj_array([p for L in layers for p in L])
    n = ctypes.c_size_t(0)
    _check(library().lora_stack_ckpt_workspace_size(arr, len(layers), n_per, ctypes.byref(n)),
           "lora_stack_ckpt_workspace_size")
    return n.value


def lora_stack_ckpt(layers, workspace, workspace_bytes, stream=None) -> None:
    """Checkpointed forward and backward of a stack of layers (see include/lora.h)."""
    n_per = len(layers[0])
    if any(len(L) != n_per for L in layers):
        raise ValueError("every layer needs the same number of projections")
    arr = _proj_array([p for L in layers for p in L])
    _check(library().lora_stack_ckpt(arr, len(layers), n_per, _ptr(workspace), int(workspace_bytes),
                                     _stream(stream)), "lora_stack_ckpt")


def make_ce_args(T, d, V, h, E, targets, loss, mask=None, topk=None, ld_topk=0, k=0, token_loss=None, dh=None,
                 vocab=None) -> lora_ce_args:
    return lora_ce_args(int(T), int(d), int(V), _ptr(h), _ptr(E), _ptr(targets), _ptr(mask), _ptr(topk),
                        int(ld_topk), int(k), _ptr(loss), _ptr(token_loss), _ptr(dh), _ptr(vocab), None)


def lora_ce_workspace_size(args: lora_ce_args) -> int:
    n = ctypes.c_size_t(0)
    _check(library().lora_ce_workspace_size(ctypes.byref(args), ctypes.byref(n)), "lora_ce_workspace_size")
    return n.value


def lora_ce_fwd_bwd(args: lora_ce_args, workspace, workspace_bytes, stream=None):
    """Reduced-vocabulary cross entropy with logits masking (see include/lora.h);
    returns (|T_set|, |J|)."""
    counts = (ctypes.c_int64 * 2)()
    args.counts = ctypes.cast(counts, ctypes.c_void_p)
    try:
        _check(library().lora_ce_fwd_bwd(ctypes.byref(args), _ptr(workspace), int(workspace_bytes), _stream(stream)),
               "lora_ce_fwd_bwd")
    finally:
        args.counts = None
    return int(counts[0]), int(counts[1])


def lora_topk_workspace_size(V: int, d: int, k: int) -> int:
    n = ctypes.c_size_t(0)
    _check(library().lora_topk_workspace_size(int(V), int(d), int(k), ctypes.byref(n)), "lora_topk_workspace_size")
    return n.value


def lora_topk_table(E, V: int, d: int, k: int, table, workspace, workspace_bytes, stream=None) -> None:
    """Top-k cosine-similarity table of the embedding E [V, d] into table [V, k] int32."""
    _check(library().lora_topk_table(_ptr(E), int(V), int(d), int(k), _ptr(table), _ptr(workspace),
                                     int(workspace_bytes), _stream(stream)), "lora_topk_table")


def lora_wait_selftest(limit_ns: int, stream=None) -> None:
    """Enqueue the bounded-wait self-check (see include/lora.h)."""
    _check(library().lora_wait_selftest(int(limit_ns), _stream(stream)), "lora_wait_selftest")


def lora_read_status(stream=None, reset: bool = True) -> int:
    st = ctypes.c_int(0)
    _check(library().lora_read_status(_stream(stream), ctypes.byref(st), 1 if reset else 0), "lora_read_status")
    return st.value


def lora_set_wait_limit_ns(ns: int) -> None:
    _check(library().lora_set_wait_limit_ns(int(ns)), "lora_set_wait_limit_ns")


def lora_launch_count() -> int:
    return int(library().lora_launch_count())


def lora_profile_begin(kinds=None) -> None:
    """Starts a profiling session over every launch group, or only the groups
    of the LORA_KERNEL_* kinds listed in `kinds`."""
    if kinds is None:
        _check(library().lora_profile_begin(), "lora_profile_begin")
    else:
        mask = 0
        for k in kinds:
            mask |= 1 << int(k)
        _check(library().lora_profile_begin_kinds(mask), "lora_profile_begin_kinds")


def lora_profile_end():
    """Returns ({kind name: device ms}, {kind name: launches}) of the session."""
    ms = (ctypes.c_double * LORA_KERNEL_KINDS)()
    n = (ctypes.c_int64 * LORA_KERNEL_KINDS)()
    _check(library().lora_profile_end(ms, n), "lora_profile_end")
    return ({KERNEL_NAMES[k]: ms[k] for k in range(LORA_KERNEL_KINDS)},
            {KERNEL_NAMES[k]: int(n[k]) for k in range(LORA_KERNEL_KINDS)})


def lora_strerror(code: int) -> str:
    return library().lora_strerror(int(code)).decode()


def lora_version() -> int:
    return library().lora_version()


def lora_last_error() -> int:
    """The code this thread's most recent library call returned (include/lora.h)."""
    return int(library().lora_last_error())
