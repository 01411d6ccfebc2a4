"""ctypes binding of include/reflex.h (argument marshalling only).

Every function keeps the C name and argument order.  Device arrays are
passed as torch tensors (their data pointers) or raw integer addresses;
`stream` defaults to torch's current CUDA stream.  All arithmetic happens in
libreflex.so; nothing here computes part of the method.
"""
from __future__ import annotations

import ctypes
from pathlib import Path

_LIB_PATH = Path(__file__).resolve().parent / "_build" / "libreflex.so"

REFLEX_OK = 0
REFLEX_EINVAL = 1
REFLEX_EKRANGE = 2
REFLEX_EWORKSPACE = 3
REFLEX_ECUDA = 4
REFLEX_ETIMEOUT = 5
REFLEX_EUNSUPPORTED = 6
REFLEX_ECAPACITY = 7

REFLEX_DTYPE_F32 = 0
REFLEX_DTYPE_BF16 = 1

REFLEX_FLAG_RENORM_TOPK = 0x1
REFLEX_FLAG_SIMT_EXPERTS = 0x2
REFLEX_FLAG_RESIDUAL = 0x4
REFLEX_FLAG_EXACT_SCORES = 0x8
REFLEX_FLAG_GATHER_IN_GEMM = 0x10
REFLEX_SIGNAL_FPS = 0
REFLEX_SIGNAL_FRONTIER = 1
REFLEX_SIGNAL_PROGRESS = 2
REFLEX_SIGNAL_CONFIDENCE = 3
REFLEX_SIGNAL_UNCERTAINTY = 4
REFLEX_RULE_REFLEX = 0
REFLEX_RULE_TOP_P = 1
REFLEX_RULE_EXPERT_THRESHOLD = 2
# the reflex_alloc_params layout above matches this ABI version
ABI_VERSION = 114
REFLEX_STAGE_ROUTE = 0x100
REFLEX_STAGE_DISPATCH = 0x200
REFLEX_STAGE_EXPERT_UP = 0x400
REFLEX_STAGE_EXPERT_DOWN = 0x800
REFLEX_STAGE_COMBINE = 0x1000

EXPORTED = (
    "reflex_default_params", "reflex_allocate", "reflex_moe_workspace_size",
    "reflex_moe_forward", "reflex_moe_status", "reflex_read_status",
    "reflex_selftest_wait_timeout", "reflex_status_string",
    "reflex_abi_version", "reflex_route_noalloc", "reflex_update_state",
    "reflex_step",
)


class reflex_alloc_params(ctypes.Structure):
    _fields_ = [("k_min", ctypes.c_int32), ("k_base", ctypes.c_int32),
                ("k_max", ctypes.c_int32), ("delta_role", ctypes.c_int32),
                ("delta_cur", ctypes.c_int32), ("q", ctypes.c_float),
                ("theta", ctypes.c_float), ("w_cf", ctypes.c_float),
                ("v_ref", ctypes.c_float), ("tau", ctypes.c_float),
                ("signal", ctypes.c_int32), ("role_shuffle", ctypes.c_int32),
                ("shuffle_seed", ctypes.c_uint64), ("count_rule", ctypes.c_int32),
                ("rule_threshold", ctypes.c_float)]


class reflex_route_record(ctypes.Structure):
    _fields_ = [("ids", ctypes.c_void_p), ("alpha", ctypes.c_void_p),
                ("counts", ctypes.c_void_p), ("offsets", ctypes.c_void_p),
                ("perm", ctypes.c_void_p), ("row_of", ctypes.c_void_p),
                ("totals", ctypes.c_void_p), ("scores", ctypes.c_void_p)]


class ReflexError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {reflex_status_string(status)} ({status})")


_lib = None


def library_path() -> Path:
    return _LIB_PATH


def load():
    """Load libreflex.so; raises if it has not been built (no fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not _LIB_PATH.exists():
        raise ImportError(
            f"{_LIB_PATH} is missing: build it with "
            "`python -m paper_2608_01784_gb300.build` (needs nvcc)")
    lib = ctypes.CDLL(str(_LIB_PATH))
    P = ctypes.c_void_p
    i32 = ctypes.c_int32
    lib.reflex_default_params.restype = None
    lib.reflex_default_params.argtypes = [ctypes.POINTER(reflex_alloc_params)]
    lib.reflex_allocate.restype = ctypes.c_int
    lib.reflex_allocate.argtypes = [P, P, P, P, P, P, P, P, i32, i32, i32,
                                    ctypes.POINTER(reflex_alloc_params), P, P, P, P]
    lib.reflex_moe_workspace_size.restype = ctypes.c_size_t
    lib.reflex_moe_workspace_size.argtypes = [i32] * 7
    lib.reflex_moe_forward.restype = ctypes.c_int
    lib.reflex_moe_forward.argtypes = [i32, P, P, P, P, P, P, i32, P, i32, i32,
                                       i32, i32, i32, ctypes.c_uint32, P,
                                       ctypes.c_size_t, P,
                                       ctypes.POINTER(reflex_route_record), P]
    lib.reflex_moe_status.restype = ctypes.c_int
    lib.reflex_moe_status.argtypes = [P, P]
    lib.reflex_read_status.restype = ctypes.c_int
    lib.reflex_read_status.argtypes = [P, P]
    lib.reflex_selftest_wait_timeout.restype = ctypes.c_int
    lib.reflex_selftest_wait_timeout.argtypes = [P, ctypes.c_uint32, P]
    lib.reflex_status_string.restype = ctypes.c_char_p
    lib.reflex_status_string.argtypes = [ctypes.c_int]
    lib.reflex_abi_version.restype = ctypes.c_int
    lib.reflex_abi_version.argtypes = []
    lib.reflex_update_state.restype = ctypes.c_int
    lib.reflex_update_state.argtypes = [P, P, P, P, P, P, P, P, P, i32, i32,
                                        ctypes.c_float, P, P, P]
    lib.reflex_step.restype = ctypes.c_int
    lib.reflex_step.argtypes = [P, P, P, P, P, P, P, i32, ctypes.POINTER(reflex_alloc_params),
                                P, P, P, i32, P, P, P, P, P, P, i32, i32, i32, i32, i32,
                                i32, ctypes.c_uint32, P, ctypes.c_size_t, P,
                                ctypes.POINTER(reflex_route_record), P]
    lib.reflex_route_noalloc.restype = ctypes.c_int
    lib.reflex_route_noalloc.argtypes = [i32, P, P, P, i32, i32, i32, i32,
                                         ctypes.c_uint32, P, P, P, P]
    if lib.reflex_abi_version() != ABI_VERSION:
        raise ImportError(f"{_LIB_PATH} has ABI version {lib.reflex_abi_version()}, "
                          f"this binding needs {ABI_VERSION}: rebuild it")
    _lib = lib
    return lib


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def reflex_status_string(status: int) -> str:
    return load().reflex_status_string(int(status)).decode()


def reflex_abi_version() -> int:
    return int(load().reflex_abi_version())


def reflex_default_params() -> reflex_alloc_params:
    p = reflex_alloc_params()
    load().reflex_default_params(ctypes.byref(p))
    return p


def make_params(**kw) -> reflex_alloc_params:
    p = reflex_default_params()
    for k, v in kw.items():
        setattr(p, k, v)
    return p


def reflex_update_state(conf_new, conf_prev1, conf_prev2, hist_len, masked,
                        block_id, seq_offsets, active_block, num_blocks, T: int,
                        B: int, theta_commit: float, committed_out=None,
                        dev_status=None, stream=None, check: bool = True) -> int:
    rc = load().reflex_update_state(
        _ptr(conf_new), _ptr(conf_prev1), _ptr(conf_prev2), _ptr(hist_len),
        _ptr(masked), _ptr(block_id), _ptr(seq_offsets), _ptr(active_block),
        _ptr(num_blocks), T, B, float(theta_commit), _ptr(committed_out),
        _ptr(dev_status), _stream(stream))
    if check and rc != REFLEX_OK:
        raise ReflexError(rc, "reflex_update_state")
    return rc


def reflex_allocate(router_scores, conf_prev1, conf_prev2, hist_len, masked,
                    block_id, seq_offsets, active_block, T: int, B: int, E: int,
                    params: reflex_alloc_params, k_out, k_sum_out=None,
                    dev_status=None, stream=None, check: bool = True) -> int:
    rc = load().reflex_allocate(
        _ptr(router_scores), _ptr(conf_prev1), _ptr(conf_prev2), _ptr(hist_len),
        _ptr(masked), _ptr(block_id), _ptr(seq_offsets), _ptr(active_block),
        T, B, E, ctypes.byref(params), _ptr(k_out), _ptr(k_sum_out),
        _ptr(dev_status), _stream(stream))
    if check and rc != REFLEX_OK:
        raise ReflexError(rc, "reflex_allocate")
    return rc


def reflex_moe_workspace_size(dtype: int, T: int, d: int, E: int, inter: int,
                              shared_inter: int, k_max: int) -> int:
    return int(load().reflex_moe_workspace_size(dtype, T, d, E, inter,
                                                shared_inter, k_max))


def reflex_moe_forward(dtype: int, hidden, w_router, w_gate_up, w_down,
                       shared_gate_up, shared_down, shared_inter: int, k,
                       T: int, d: int, E: int, inter: int, k_max: int,
                       flags: int, workspace, ws_bytes: int, out,
                       rec: reflex_route_record | None = None, stream=None,
                       check: bool = True) -> int:
    rc = load().reflex_moe_forward(
        dtype, _ptr(hidden), _ptr(w_router), _ptr(w_gate_up), _ptr(w_down),
        _ptr(shared_gate_up), _ptr(shared_down), shared_inter, _ptr(k), T, d,
        E, inter, k_max, flags, _ptr(workspace), ws_bytes, _ptr(out),
        ctypes.byref(rec) if rec is not None else None, _stream(stream))
    if check and rc != REFLEX_OK:
        raise ReflexError(rc, "reflex_moe_forward")
    return rc


def reflex_step(conf_prev1, conf_prev2, hist_len, masked, block_id, seq_offsets,
                active_block, B: int, params: reflex_alloc_params, k_out, k_sum_out,
                alloc_status, dtype: int, hidden, w_router, w_gate_up, w_down,
                shared_gate_up, shared_down, shared_inter: int, T: int, d: int, E: int,
                inter: int, k_max: int, flags: int, workspace, ws_bytes: int, out,
                rec: reflex_route_record | None = None, stream=None,
                check: bool = True) -> int:
    rc = load().reflex_step(
        _ptr(conf_prev1), _ptr(conf_prev2), _ptr(hist_len), _ptr(masked), _ptr(block_id),
        _ptr(seq_offsets), _ptr(active_block), B, ctypes.byref(params), _ptr(k_out),
        _ptr(k_sum_out), _ptr(alloc_status), dtype, _ptr(hidden), _ptr(w_router),
        _ptr(w_gate_up), _ptr(w_down), _ptr(shared_gate_up), _ptr(shared_down),
        shared_inter, T, d, E, inter, k_max, flags, _ptr(workspace), ws_bytes, _ptr(out),
        ctypes.byref(rec) if rec is not None else None, _stream(stream))
    if check and rc != REFLEX_OK:
        raise ReflexError(rc, "reflex_step")
    return rc


def reflex_moe_status(workspace, stream=None) -> int:
    return int(load().reflex_moe_status(_ptr(workspace), _stream(stream)))


def reflex_read_status(dev_status, stream=None) -> int:
    return int(load().reflex_read_status(_ptr(dev_status), _stream(stream)))


def reflex_selftest_wait_timeout(dev_status, limit_us: int, stream=None) -> int:
    return int(load().reflex_selftest_wait_timeout(_ptr(dev_status), limit_us,
                                                   _stream(stream)))


REFLEX_NOALLOC_MAX_SCORES = 1 << 20


def reflex_route_noalloc(dtype: int, hidden, w_router, k, T: int, d: int,
                         E: int, k_max: int, flags: int, ids_out, alpha_out,
                         dev_status=None, stream=None) -> int:
    """Routing step with no device allocation (scratch in the library's own
    fixed array; see include/reflex.h)."""
    return int(load().reflex_route_noalloc(
        dtype, _ptr(hidden), _ptr(w_router), _ptr(k), T, d, E, k_max, flags,
        _ptr(ids_out), _ptr(alpha_out), _ptr(dev_status), _stream(stream)))
