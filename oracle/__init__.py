"""Plain CPU oracle for the REFLEX per-forward MoE path (test infrastructure).

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The
product path (``paper_2608_01784_gb300``) never imports it and shares no code
with it.

The arithmetic lives in ``reflex_oracle.c`` (plain C, ``-ffp-contract=off``);
this module compiles it with gcc and marshals numpy arrays into it.  The C
file's header lists which paper passage each function follows:

* ``allocate``        Refinement-Role Budgeting (Eq. 5) + Frontier-Guided
                      Expert Reallocation (forecast, Eq. 6-8, Eq. 9) + clip.
* ``router_logits``   router scores of Sec. 3.2 (sequential fp32 fma chain).
* ``select``          TopK of Eq. 2 and the normalised router weight.
* ``rule_counts``     the Top-p and Expert-Threshold counts of the
                      threshold-based comparison methods (App. B).
* ``permutation``     (expert, token)-ordered pair list that executes Eq. 2.
* ``moe_tokens``      Eq. 2 with SwiGLU experts (+ shared expert), fp64.
* ``moe_stack``       a stack of such layers with the residual update
                      h <- bf16(h + MoE(h)), the per-token counts shared by
                      every layer (Sec. 3.3).

Parity unpinned: none of the functions above (see tests/test_oracle_pins.py);
the paper-level AvgK / pair-reduction numbers of Table 1 need the paper's
models and data and are not reproduced.
"""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
_SRC = _HERE / "reflex_oracle.c"
_BUILD = _HERE / "_build"
_LIB_PATH = _BUILD / "liboracle.so"
_lib = None


def build(force: bool = False) -> Path:
    """Compile reflex_oracle.c into oracle/_build/liboracle.so (gcc, -O2,
    -ffp-contract=off, OpenMP when available)."""
    _BUILD.mkdir(exist_ok=True)
    if (not force and _LIB_PATH.exists()
            and _LIB_PATH.stat().st_mtime >= _SRC.stat().st_mtime):
        return _LIB_PATH
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        raise RuntimeError("oracle build needs gcc")
    tmp = _BUILD / f"liboracle.{os.getpid()}.so"
    base = [cc, "-O2", "-ffp-contract=off", "-fno-fast-math", "-std=c11",
            "-fPIC", "-shared", str(_SRC), "-o", str(tmp), "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(str(build()))
    p = ctypes.c_void_p
    i32 = ctypes.c_int32
    f32 = ctypes.c_float
    lib.oracle_exp_f32.restype = f32
    lib.oracle_exp_f32.argtypes = [f32]
    lib.oracle_exp_f32_n.restype = None
    lib.oracle_exp_f32_n.argtypes = [p, p, ctypes.c_int64]
    lib.oracle_fps.restype = f32
    lib.oracle_fps.argtypes = [f32, f32, i32, f32, f32, f32, f32]
    lib.oracle_fps_n.restype = None
    lib.oracle_fps_n.argtypes = [p, p, p, ctypes.c_int64, f32, f32, f32, f32, p]
    lib.oracle_allocate.restype = ctypes.c_int
    lib.oracle_allocate.argtypes = [p, p, p, p, p, p, p, i32, i32,
                                    i32, i32, i32, i32, i32,
                                    f32, f32, f32, f32, f32, p, p]
    lib.oracle_allocate_ex.restype = ctypes.c_int
    lib.oracle_allocate_ex.argtypes = [p, p, p, p, p, p, p, i32, i32,
                                       i32, i32, i32, i32, i32,
                                       f32, f32, f32, f32, f32,
                                       i32, i32, ctypes.c_uint64, p, p]
    lib.oracle_update_state.restype = ctypes.c_int
    lib.oracle_update_state.argtypes = [p, p, p, p, p, p, p, p, p, i32, i32, f32, p]
    lib.oracle_rank_key.restype = f32
    lib.oracle_rank_key.argtypes = [i32, f32, f32, i32, f32, f32, f32, f32]
    lib.oracle_splitmix64.restype = ctypes.c_uint64
    lib.oracle_splitmix64.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
    lib.oracle_router_logits.restype = None
    lib.oracle_router_logits.argtypes = [i32, p, p, i32, i32, i32, p]
    lib.oracle_select.restype = ctypes.c_int
    lib.oracle_select.argtypes = [p, p, i32, i32, i32, i32, p, p]
    lib.oracle_rule_counts.restype = ctypes.c_int
    lib.oracle_rule_counts.argtypes = [p, i32, i32, i32, f32, i32, i32, p]
    lib.oracle_permutation.restype = ctypes.c_int64
    lib.oracle_permutation.argtypes = [p, p, i32, i32, i32, p, p, p]
    lib.oracle_moe_tokens.restype = None
    lib.oracle_moe_tokens.argtypes = [i32, p, p, p, p, p, i32, p, p, p, p,
                                      i32, i32, i32, i32, p]
    lib.oracle_num_threads.restype = ctypes.c_int
    lib.oracle_num_threads.argtypes = []
    lib.oracle_set_num_threads.restype = None
    lib.oracle_set_num_threads.argtypes = [ctypes.c_int]
    lib.oracle_bf16_from_f64_n.restype = None
    lib.oracle_bf16_from_f64_n.argtypes = [p, ctypes.c_int64, p]
    lib.oracle_residual_bf16.restype = None
    lib.oracle_residual_bf16.argtypes = [p, p, ctypes.c_int64, p]
    _lib = lib
    return lib


def _ptr(a: np.ndarray | None):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"], "oracle arrays must be C-contiguous"
    return a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def set_num_threads(n: int) -> None:
    """Threads of the oracle's OpenMP loops from now on."""
    _load().oracle_set_num_threads(int(n))


def exp_f32(x) -> np.ndarray:
    x = _c(x, np.float32).ravel()
    y = np.empty_like(x)
    _load().oracle_exp_f32_n(_ptr(x), _ptr(y), x.size)
    return y


def fps(c1, c2, hist, theta, w_cf, v_ref, tau) -> np.ndarray:
    c1 = _c(c1, np.float32).ravel()
    c2 = _c(c2, np.float32).ravel()
    hist = _c(hist, np.uint8).ravel()
    s = np.empty_like(c1)
    _load().oracle_fps_n(_ptr(c1), _ptr(c2), _ptr(hist), c1.size, theta, w_cf,
                         v_ref, tau, _ptr(s))
    return s


def allocate(conf1, conf2, hist_len, masked, block_id, seq_offsets,
             active_block, *, k_min, k_base, k_max, delta_role, delta_cur,
             q, theta, w_cf, v_ref, tau, signal: int = 0, role_shuffle: int = 0,
             shuffle_seed: int = 0, return_scores: bool = False):
    """Per-token expert counts of REFLEX (Eq. 5, Eq. 9, clip); int32 [T].
    signal / role_shuffle / shuffle_seed select the App. C ablations (rank
    key of the Eq. 9 groups; Role-Shuffled RRB)."""
    conf1 = _c(conf1, np.float32)
    conf2 = _c(conf2, np.float32)
    hist_len = _c(hist_len, np.uint8)
    masked = _c(masked, np.uint8)
    block_id = _c(block_id, np.int32)
    seq_offsets = _c(seq_offsets, np.int32)
    active_block = _c(active_block, np.int32)
    T = block_id.size
    B = active_block.size
    k = np.empty(T, np.int32)
    s = np.empty(T, np.float32)
    rc = _load().oracle_allocate_ex(
        _ptr(conf1), _ptr(conf2), _ptr(hist_len), _ptr(masked),
        _ptr(block_id), _ptr(seq_offsets), _ptr(active_block), T, B,
        k_min, k_base, k_max, delta_role, delta_cur, q, theta, w_cf, v_ref,
        tau, int(signal), int(role_shuffle), int(shuffle_seed) & (2**64 - 1),
        _ptr(k), _ptr(s))
    if rc != 0:
        raise ValueError("oracle_allocate: invalid input")
    return (k, s) if return_scores else k


def update_state(state: dict, conf_new, num_blocks, theta_commit: float):
    """Block-wise inference after one forward (Sec. 3.1, Eq. 1) on a numpy
    state dict: returns (new state dict, committed per sequence)."""
    st = {k: np.array(v, copy=True) for k, v in state.items()}
    st["conf1"] = _c(st["conf1"], np.float32)
    st["conf2"] = _c(st["conf2"], np.float32)
    st["hist_len"] = _c(st["hist_len"], np.uint8)
    st["masked"] = _c(st["masked"], np.uint8)
    st["active_block"] = _c(st["active_block"], np.int32)
    conf_new = _c(conf_new, np.float32)
    block_id = _c(st["block_id"], np.int32)
    seq_off = _c(st["seq_offsets"], np.int32)
    nb = _c(num_blocks, np.int32)
    T = block_id.size
    B = st["active_block"].size
    committed = np.zeros(B, np.int32)
    rc = _load().oracle_update_state(
        _ptr(conf_new), _ptr(st["conf1"]), _ptr(st["conf2"]), _ptr(st["hist_len"]),
        _ptr(st["masked"]), _ptr(block_id), _ptr(seq_off), _ptr(st["active_block"]),
        _ptr(nb), T, B, theta_commit, _ptr(committed))
    if rc != 0:
        raise ValueError("oracle_update_state: invalid input")
    return st, committed


def rank_key(signal: int, c1: float, c2: float, hist: int, theta: float,
             w_cf: float, v_ref: float, tau: float) -> float:
    """Rank key of one J_h member under an App. C signal (0 FPS, 1 F, 2 P,
    3 c^{t-1}, 4 1 - c^{t-1})."""
    return float(_load().oracle_rank_key(signal, c1, c2, hist, theta, w_cf, v_ref, tau))


def splitmix64(seed: int, n: int) -> int:
    """Output number n (n >= 1) of the splitmix64 stream seeded with seed."""
    return int(_load().oracle_splitmix64(seed & (2**64 - 1), n & (2**64 - 1)))


def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return 0
    if a.dtype == np.uint16:  # bf16 bit patterns
        return 1
    raise TypeError("oracle inputs are float32 or bf16 bits (uint16)")


def router_logits(hidden: np.ndarray, w_router: np.ndarray) -> np.ndarray:
    """z[T, E] fp32 by the sequential fma chain over the hidden index."""
    hidden = np.ascontiguousarray(hidden)
    w_router = np.ascontiguousarray(w_router)
    dt = _dtype_code(hidden)
    assert _dtype_code(w_router) == dt
    T, d = hidden.shape
    E = w_router.shape[0]
    z = np.empty((T, E), np.float32)
    _load().oracle_router_logits(dt, _ptr(hidden), _ptr(w_router), T, d, E,
                                 _ptr(z))
    return z


def select(z: np.ndarray, k: np.ndarray, k_max: int, renorm: bool = True):
    """(ids int32 [T, k_max], alpha fp64 [T, k_max])."""
    z = _c(z, np.float32)
    k = _c(k, np.int32)
    T, E = z.shape
    ids = np.empty((T, k_max), np.int32)
    alpha = np.empty((T, k_max), np.float64)
    rc = _load().oracle_select(_ptr(z), _ptr(k), T, E, k_max, int(renorm),
                               _ptr(ids), _ptr(alpha))
    if rc != 0:
        raise ValueError("oracle_select: some k_t outside [1, min(k_max, E)]")
    return ids, alpha


RULE_TOP_P = 1
RULE_EXPERT_THRESHOLD = 2


def rule_counts(z: np.ndarray, rule: int, threshold: float, k_min: int = 1,
                k_max: int = 12) -> np.ndarray:
    """Counts of the threshold-based comparison methods (App. B) from router
    scores z [T, E]: rule 1 = Top-p (threshold p), 2 = Expert-Threshold
    routing; clipped to [k_min, min(k_max, E)].  int32 [T]."""
    z = _c(z, np.float32)
    T, E = z.shape
    k = np.empty(T, np.int32)
    rc = _load().oracle_rule_counts(_ptr(z), T, E, int(rule), float(threshold),
                                    int(k_min), int(k_max), _ptr(k))
    if rc != 0:
        raise ValueError("oracle_rule_counts: invalid rule or bounds")
    return k


def permutation(ids: np.ndarray, k: np.ndarray, E: int):
    """(offsets int32 [E+1], perm int32 [sum k], row_of int32 [T, k_max])."""
    ids = _c(ids, np.int32)
    k = _c(k, np.int32)
    T, k_max = ids.shape
    offsets = np.empty(E + 1, np.int32)
    perm = np.empty(max(int(k.sum()), 1), np.int32)
    row_of = np.empty((T, k_max), np.int32)
    n = _load().oracle_permutation(_ptr(ids), _ptr(k), T, E, k_max,
                                   _ptr(offsets), _ptr(perm), _ptr(row_of))
    return offsets, perm[:n].copy(), row_of


def moe_tokens(hidden, w_gate_up, w_down, ids, alpha, k, tokens, *,
               shared_gate_up=None, shared_down=None) -> np.ndarray:
    """Eq. 2 (+ shared expert) for the listed tokens; fp64 [len(tokens), d]."""
    hidden = np.ascontiguousarray(hidden)
    w_gate_up = np.ascontiguousarray(w_gate_up)
    w_down = np.ascontiguousarray(w_down)
    dt = _dtype_code(hidden)
    T, d = hidden.shape
    inter = w_down.shape[-1]
    ids = _c(ids, np.int32)
    alpha = _c(alpha, np.float64)
    k = _c(k, np.int32)
    tokens = _c(tokens, np.int32)
    k_max = ids.shape[1]
    s_inter = 0
    if shared_gate_up is not None:
        shared_gate_up = np.ascontiguousarray(shared_gate_up)
        shared_down = np.ascontiguousarray(shared_down)
        s_inter = shared_down.shape[-1]
    out = np.empty((tokens.size, d), np.float64)
    _load().oracle_moe_tokens(dt, _ptr(hidden), _ptr(w_gate_up), _ptr(w_down),
                              _ptr(shared_gate_up), _ptr(shared_down), s_inter,
                              _ptr(ids), _ptr(alpha), _ptr(k), _ptr(tokens),
                              tokens.size, d, inter, k_max, _ptr(out))
    return out


def moe_layer(hidden, w_router, w_gate_up, w_down, k, k_max, *, tokens=None,
              renorm=True, shared_gate_up=None, shared_down=None) -> dict:
    """Whole layer in the paper's order: scores -> TopK/alpha -> pairs ->
    Eq. 2 for ``tokens`` (all tokens when None)."""
    E = w_router.shape[0]
    z = router_logits(hidden, w_router)
    ids, alpha = select(z, k, k_max, renorm)
    offsets, perm, row_of = permutation(ids, k, E)
    if tokens is None:
        tokens = np.arange(hidden.shape[0], dtype=np.int32)
    out = moe_tokens(hidden, w_gate_up, w_down, ids, alpha, k, tokens,
                     shared_gate_up=shared_gate_up, shared_down=shared_down)
    return dict(z=z, ids=ids, alpha=alpha, offsets=offsets, perm=perm,
                row_of=row_of, tokens=np.asarray(tokens, np.int32), out=out)


def bf16_from_f64(x) -> np.ndarray:
    """Round fp64 values to bf16 (nearest, ties to even); uint16 bits."""
    x = _c(x, np.float64)
    out = np.empty(x.shape, np.uint16)
    _load().oracle_bf16_from_f64_n(_ptr(x), x.size, _ptr(out))
    return out


def residual_bf16(h_bits: np.ndarray, out: np.ndarray) -> np.ndarray:
    """bf16(h + out) for bf16 bits h and an fp64 layer output."""
    h_bits = _c(h_bits, np.uint16)
    out = _c(out, np.float64)
    assert h_bits.shape == out.shape
    nxt = np.empty_like(h_bits)
    _load().oracle_residual_bf16(_ptr(h_bits), _ptr(out), h_bits.size, _ptr(nxt))
    return nxt


def moe_stack(hidden_bits: np.ndarray, layers: list, k, k_max: int,
              renorm: bool = True) -> list:
    """Layer by layer: res_l = Eq. 2 on h_l with layer l's weights and the
    shared counts k; h_{l+1} = bf16(h_l + res_l.out).  Returns one dict per
    layer with its input h (bf16 bits), routing record and output h."""
    h = np.ascontiguousarray(hidden_bits, np.uint16)
    trace = []
    for lay in layers:
        res = moe_layer(h, lay["w_router"], lay["w_gate_up"], lay["w_down"], k,
                        k_max, renorm=renorm,
                        shared_gate_up=lay.get("shared_gate_up"),
                        shared_down=lay.get("shared_down"))
        nxt = residual_bf16(h, res["out"])
        res["h_in"] = h
        res["h_out"] = nxt
        trace.append(res)
        h = nxt
    return trace
