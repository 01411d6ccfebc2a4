"""Seeded synthetic inputs for the REFLEX MoE hot path.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic, so both the CUDA path and the CPU oracle can be fed from
it.  Every array is a pure function of (config, seed).

Workload shapes (d, E, inter, shared expert, K bounds) follow the two model
families the paper evaluates (LLaDA-MoE and LLaDA2.0-mini, Sec. 5.1) and the
hyper-parameters of Sec. 5.1 (theta = 0.9, K_base = 8, delta_role = 4,
delta_cur = 2, q = 0.25, v_ref = 0.01, tau = 0.05, w_cf = 0.30 / 0.25,
block length 32).  The paper's datasets and checkpoints are not used: hidden
states, router and expert weights, confidences and mask states are synthetic.

Recipe (all streams are numpy PCG64 seeded from (seed, stream name)):
  hidden       N(0, 1)
  weights      N(0, std): std = 1/sqrt(fan_in) for the tiny fp32 case,
               0.02 otherwise; bf16 storage rounds to nearest even.
  layout       n_seq sequences of prompt_len prompt tokens (block 0) followed
               by gen_len target tokens in blocks of `block`.
  active block per sequence: given, or uniform over 1..Q from the seed.
  masks        "half":      a seeded half of the target tokens is masked;
               "linear":    target block j of Q has masked fraction (j-1)/(Q-1);
               "blockwise": blocks before the active one are resolved, the
                            active one has a U(0,1) masked fraction, blocks
                            after it are fully masked (block-wise decoding,
                            Eq. 1).
  confidences  c^{t-1}: U(0,1) ("uniform") or Beta(2,2) on masked and
               Beta(5,1) on resolved positions ("beta");
               c^{t-2} = clip(c^{t-1} - u, 0, 1), u ~ U(-0.2, 0.2), so lagged
               changes straddle +-w_cf/2; hist_len = 2 unless overridden.
"""
from __future__ import annotations

import dataclasses
import zlib
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import torch

_CHUNK = 1 << 22


@dataclasses.dataclass(frozen=True)
class LayerConfig:
    name: str
    dtype: str                 # "f32" or "bf16" storage
    d: int
    E: int
    inter: int
    shared_inter: int
    k_min: int
    k_base: int
    k_max: int
    delta_role: int
    delta_cur: int
    w_cf: float
    n_seq: int
    prompt_len: int
    gen_len: int
    block: int
    weight_std: float | None   # None: 1/sqrt(fan_in)
    conf: str                  # "uniform" | "beta"
    mask_rule: str             # "half" | "linear" | "blockwise"
    active: int | None = None  # fixed active block, or None for seeded
    q: float = 0.25
    theta: float = 0.9
    v_ref: float = 0.01
    tau: float = 0.05
    description: str = ""

    @property
    def seq_len(self) -> int:
        return self.prompt_len + self.gen_len

    @property
    def T(self) -> int:
        return self.n_seq * self.seq_len

    @property
    def n_blocks(self) -> int:
        return self.gen_len // self.block

    def alloc_params(self, **override) -> dict:
        p = dict(k_min=self.k_min, k_base=self.k_base, k_max=self.k_max,
                 delta_role=self.delta_role, delta_cur=self.delta_cur,
                 q=self.q, theta=self.theta, w_cf=self.w_cf, v_ref=self.v_ref,
                 tau=self.tau)
        p.update(override)
        return p

    def with_(self, **kw) -> "LayerConfig":
        return dataclasses.replace(self, **kw)


CONFIGS: dict[str, LayerConfig] = {
    # tiny fp32 layer the oracle finishes instantly
    "tiny_fp32": LayerConfig(
        name="tiny_fp32", dtype="f32", d=256, E=8, inter=128, shared_inter=0,
        k_min=1, k_base=2, k_max=4, delta_role=1, delta_cur=1, w_cf=0.30,
        n_seq=1, prompt_len=32, gen_len=64, block=32, weight_std=None,
        conf="uniform", mask_rule="half", active=2,
        description="T=96 (32 prompt + 2 blocks of 32, second active), d=256, "
                    "E=8, inter=128, K in [1,4], fp32"),
    # LLaDA-MoE-shaped layer
    "llada_moe": LayerConfig(
        name="llada_moe", dtype="bf16", d=2048, E=64, inter=1024,
        shared_inter=0, k_min=2, k_base=8, k_max=12, delta_role=4,
        delta_cur=2, w_cf=0.30, n_seq=1, prompt_len=512, gen_len=512,
        block=32, weight_std=0.02, conf="beta", mask_rule="linear",
        description="LLaDA-MoE-shaped layer: T=1024 (512 prompt + 512 gen, "
                    "block 32), d=2048, E=64, inter=1024, K in [2,12], bf16"),
    # LLaDA2.0-mini-shaped layer with a shared expert
    "llada2_mini": LayerConfig(
        name="llada2_mini", dtype="bf16", d=2048, E=256, inter=512,
        shared_inter=512, k_min=2, k_base=8, k_max=12, delta_role=4,
        delta_cur=2, w_cf=0.25, n_seq=8, prompt_len=256, gen_len=768,
        block=32, weight_std=0.02, conf="beta", mask_rule="blockwise",
        description="LLaDA2.0-mini-shaped layer: 8 x 1024 tokens (256 prompt "
                    "+ 768 gen, block 32), d=2048, E=256 + 1 shared expert, "
                    "inter=512, K in [2,12], bf16"),
    # one layer of the 16-layer stack: LLaDA-MoE shapes, batch 32 x 1024
    "llada_moe_b32": LayerConfig(
        name="llada_moe_b32", dtype="bf16", d=2048, E=64, inter=1024,
        shared_inter=0, k_min=2, k_base=8, k_max=12, delta_role=4,
        delta_cur=2, w_cf=0.30, n_seq=32, prompt_len=512, gen_len=512,
        block=32, weight_std=0.02, conf="beta", mask_rule="blockwise",
        description="one layer of a 16-layer LLaDA-MoE-shaped stack, batch "
                    "32 x 1024 tokens, bf16"),
}


def _seed_for(seed: int, stream: str) -> np.random.SeedSequence:
    return np.random.SeedSequence([int(seed) & 0xFFFFFFFF,
                                   zlib.crc32(stream.encode())])


def _rng(seed: int, stream: str) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(_seed_for(seed, stream)))


def normal_f32(seed: int, stream: str, n: int, std: float) -> np.ndarray:
    """n draws of N(0, std^2) as float32, in fixed 4M-element chunks (one
    child stream per chunk, so the values do not depend on thread count)."""
    out = np.empty(n, dtype=np.float32)
    nch = (n + _CHUNK - 1) // _CHUNK
    kids = _seed_for(seed, stream).spawn(max(nch, 1))

    def work(i):
        g = np.random.Generator(np.random.PCG64(kids[i]))
        lo = i * _CHUNK
        hi = min(n, lo + _CHUNK)
        g.standard_normal(hi - lo, dtype=np.float32, out=out[lo:hi])
        out[lo:hi] *= np.float32(std)

    if nch <= 1:
        if n:
            work(0)
    else:
        with ThreadPoolExecutor(min(16, nch)) as ex:
            list(ex.map(work, range(nch)))
    return out


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest, ties to even); returns uint16 bits."""
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32)


def _weights(cfg: LayerConfig, seed: int, stream: str, shape, fan_in: int):
    std = cfg.weight_std if cfg.weight_std is not None else 1.0 / np.sqrt(fan_in)
    n = int(np.prod(shape))
    w = normal_f32(seed, stream, n, std).reshape(shape)
    return to_bf16_bits(w) if cfg.dtype == "bf16" else w


def make_state(cfg: LayerConfig, seed: int = 0, hist_len: int | None = None,
               T: int | None = None) -> dict:
    """Refinement state of one denoising forward: block ids, sequence
    offsets, active block per sequence, mask, confidence history.

    ``T`` (optional) truncates/extends the batch to whole sequences of the
    config's layout (used by token-count sweeps)."""
    n_seq = cfg.n_seq if T is None else max(1, T // cfg.seq_len)
    Q = cfg.n_blocks
    L = cfg.seq_len
    block_id = np.zeros(n_seq * L, np.int32)
    for s in range(n_seq):
        base = s * L + cfg.prompt_len
        block_id[base:base + cfg.gen_len] = 1 + np.arange(cfg.gen_len) // cfg.block
    seq_offsets = (np.arange(n_seq + 1, dtype=np.int32) * L).astype(np.int32)
    g = _rng(seed, "active")
    if cfg.active is not None:
        active = np.full(n_seq, cfg.active, np.int32)
    else:
        active = g.integers(1, Q + 1, size=n_seq).astype(np.int32)
    gm = _rng(seed, "mask")
    masked = np.zeros(n_seq * L, np.uint8)
    for s in range(n_seq):
        base = s * L + cfg.prompt_len
        for j in range(1, Q + 1):
            lo = base + (j - 1) * cfg.block
            hi = lo + cfg.block
            if cfg.mask_rule == "half":
                continue
            if cfg.mask_rule == "linear":
                frac = (j - 1) / max(Q - 1, 1)
            elif cfg.mask_rule == "blockwise":
                a = int(active[s])
                frac = 0.0 if j < a else (1.0 if j > a else float(gm.uniform()))
            else:
                raise ValueError(cfg.mask_rule)
            nm = int(round(frac * cfg.block))
            sel = gm.permutation(cfg.block)[:nm]
            masked[lo + sel] = 1
        if cfg.mask_rule == "half":
            sel = gm.permutation(cfg.gen_len)[: cfg.gen_len // 2]
            masked[base + sel] = 1
    gc = _rng(seed, "conf")
    n = n_seq * L
    if cfg.conf == "uniform":
        conf1 = gc.uniform(size=n).astype(np.float32)
    else:
        a = gc.beta(2.0, 2.0, size=n)
        b = gc.beta(5.0, 1.0, size=n)
        conf1 = np.where(masked == 1, a, b).astype(np.float32)
    u = gc.uniform(-0.2, 0.2, size=n)
    conf2 = np.clip(conf1.astype(np.float64) - u, 0.0, 1.0).astype(np.float32)
    hl = np.full(n, 2 if hist_len is None else hist_len, np.uint8)
    return dict(block_id=block_id, seq_offsets=seq_offsets, active_block=active,
                masked=masked, conf1=conf1, conf2=conf2, hist_len=hl)


def layer_weights(cfg: LayerConfig, seed: int = 0, prefix: str = "") -> dict:
    """Router and expert weights of one MoE layer (no hidden states); the
    streams are named `prefix` + array name, so each layer of a stack draws
    its own weights from the same seed."""
    d, E, I = cfg.d, cfg.E, cfg.inter
    out = {}
    out["w_router"] = _weights(cfg, seed, prefix + "w_router", (E, d), d)
    out["w_gate_up"] = _weights(cfg, seed, prefix + "w_gate_up", (E, 2 * I, d), d)
    out["w_down"] = _weights(cfg, seed, prefix + "w_down", (E, d, I), I)
    if cfg.shared_inter:
        S = cfg.shared_inter
        out["shared_gate_up"] = _weights(cfg, seed, prefix + "shared_gate_up", (2 * S, d), d)
        out["shared_down"] = _weights(cfg, seed, prefix + "shared_down", (d, S), S)
    return out


def make_hidden(cfg: LayerConfig, seed: int = 0, T: int | None = None) -> np.ndarray:
    """Hidden states [T, d] ~ N(0, 1) (bf16 bits for bf16 layers)."""
    T = cfg.T if T is None else T
    h = normal_f32(seed, "hidden", T * cfg.d, 1.0).reshape(T, cfg.d)
    return to_bf16_bits(h) if cfg.dtype == "bf16" else h


def make_layer(cfg: LayerConfig, seed: int = 0, T: int | None = None) -> dict:
    """Hidden states and weights of one MoE layer.

    Layouts (row-major): hidden [T, d]; w_router [E, d];
    w_gate_up [E, 2*inter, d] (rows [0, inter) gate, [inter, 2*inter) up);
    w_down [E, d, inter]; shared_gate_up [2*s, d]; shared_down [d, s].
    bf16 arrays are uint16 bit patterns."""
    out = dict(hidden=make_hidden(cfg, seed, T))
    out.update(layer_weights(cfg, seed))
    return out


def make_stack(cfg: LayerConfig, seed: int = 0, n_layers: int = 16,
               T: int | None = None) -> dict:
    """A stack of `n_layers` MoE layers of one shape: the first layer's input
    hidden states and, per layer l, its own router and expert weights (streams
    "layer{l}/..." of the seed).  Returns {"hidden": [T, d], "layers": [...]}."""
    return dict(hidden=make_hidden(cfg, seed, T),
                layers=[layer_weights(cfg, seed, f"layer{l}/") for l in range(n_layers)])


def skewed_k(T: int, skew: float, k_min: int, k_base: int, k_max: int,
             seed: int = 0) -> np.ndarray:
    """Synthetic count vector for skew sweeps: a fraction 0.7*skew of tokens
    gets k_min, 0.3*skew gets k_max, the rest k_base, in seeded order."""
    n_lo = int(round(0.7 * skew * T))
    n_hi = int(round(0.3 * skew * T))
    k = np.full(T, k_base, np.int32)
    k[:n_lo] = k_min
    k[n_lo:n_lo + n_hi] = k_max
    return _rng(seed, "skew").permutation(k).astype(np.int32)


def sample_tokens(state: dict, stride: int = 61) -> np.ndarray:
    """Token subsample for large-size checks: every active-block token plus
    every `stride`-th token."""
    T = state["block_id"].size
    act = np.zeros(T, bool)
    for s in range(state["active_block"].size):
        lo, hi = state["seq_offsets"][s], state["seq_offsets"][s + 1]
        act[lo:hi] = state["block_id"][lo:hi] == state["active_block"][s]
    act[::stride] = True
    return np.nonzero(act)[0].astype(np.int32)
