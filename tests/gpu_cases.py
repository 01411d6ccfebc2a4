"""Shared drivers for the GPU parity tests: run the CUDA path through the C ABI
and the oracle on the same seeded inputs.  Oracle calls stay on the host;
nothing the GPU produces is fed to the oracle."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2608_01784_gb300 import _binding as B
from paper_2608_01784_gb300 import api
from paper_2608_01784_gb300 import workloads as W

# Layer-output tolerance for bf16 storage with fp32 accumulation.
BF16_REL_L2 = 1e-2
BF16_MAX_ABS = 2e-2
# fp32 storage: fp32 accumulation against the fp64 oracle.
F32_REL_L2 = 1e-5
F32_MAX_ABS = 1e-4
ALPHA_RTOL = 2e-5


def bf16_ulp(x) -> np.ndarray:
    """Spacing of bf16 numbers (8 significant bits) at |x|: 2^(floor(log2|x|) - 7)."""
    ax = np.maximum(np.abs(np.asarray(x, np.float64)), 2.0 ** -126)
    return np.exp2(np.floor(np.log2(ax)) - 7)


def residual_excess(gpu: np.ndarray, ref: np.ndarray, rounded_ref: bool) -> float:
    """Largest |gpu - ref| beyond what the bf16 rounding of a residual output
    h + MoE(h) allows on top of the MoE term's BF16_MAX_ABS; <= 0 passes.

    The layer output is rounded to bf16 once, after the residual sum.  Against
    an unrounded (fp64) reference that rounding adds at most half a bf16 ulp
    of the sum; against a reference rounded to bf16 itself the two sums may
    round to neighbouring values, one ulp apart.  The ulp is taken at the
    larger of the two magnitudes (a sum just below a power of two may round up
    to it)."""
    g = gpu.astype(np.float64)
    u = bf16_ulp(np.maximum(np.abs(g), np.abs(ref)))
    allow = BF16_MAX_ABS + (u if rounded_ref else 0.5 * u)
    return float((np.abs(g - ref) - allow).max())


def params_of(cfg: W.LayerConfig, **override) -> B.reflex_alloc_params:
    return B.make_params(**cfg.alloc_params(**override))


def gpu_allocate(state: dict, p: B.reflex_alloc_params):
    dstate = api.state_to_device(state)
    k, ksum, status = api.allocate(dstate, p)
    torch.cuda.synchronize()
    return (k.cpu().numpy(), int(ksum.item()),
            B.reflex_read_status(status))


def oracle_allocate(state: dict, p: B.reflex_alloc_params):
    return oracle.allocate(state["conf1"], state["conf2"], state["hist_len"],
                           state["masked"], state["block_id"],
                           state["seq_offsets"], state["active_block"],
                           k_min=p.k_min, k_base=p.k_base, k_max=p.k_max,
                           delta_role=p.delta_role, delta_cur=p.delta_cur,
                           q=p.q, theta=p.theta, w_cf=p.w_cf, v_ref=p.v_ref,
                           tau=p.tau, signal=p.signal, role_shuffle=p.role_shuffle,
                           shuffle_seed=p.shuffle_seed)


def to_f32(x: torch.Tensor) -> np.ndarray:
    return x.float().cpu().numpy()


class GpuLayer:
    """Device copy of a host layer plus a MoELayer sized for it."""

    def __init__(self, cfg: W.LayerConfig, layer: dict, T: int | None = None):
        self.cfg = cfg
        self.host = layer
        self.dev = api.layer_to_device(layer, cfg.dtype)
        T = layer["hidden"].shape[0] if T is None else T
        self.moe = api.MoELayer(self.dev, dtype=cfg.dtype, d=cfg.d, E=cfg.E,
                                inter=cfg.inter, shared_inter=cfg.shared_inter,
                                k_max=cfg.k_max, max_tokens=T)

    def forward(self, k: np.ndarray, flags=B.REFLEX_FLAG_RENORM_TOPK,
                hidden: torch.Tensor | None = None):
        kd = torch.from_numpy(np.ascontiguousarray(k, np.int32)).cuda()
        h = self.dev["hidden"] if hidden is None else hidden
        out = self.moe.forward(h, kd, flags=flags)
        torch.cuda.synchronize()
        status = self.moe.status()
        rec = {k: v.cpu().numpy() for k, v in self.moe.record().items()}
        return to_f32(out), rec, status


def oracle_layer(cfg: W.LayerConfig, layer: dict, k: np.ndarray, tokens=None,
                 renorm=True):
    return oracle.moe_layer(layer["hidden"], layer["w_router"],
                            layer["w_gate_up"], layer["w_down"], k, cfg.k_max,
                            tokens=tokens, renorm=renorm,
                            shared_gate_up=layer.get("shared_gate_up"),
                            shared_down=layer.get("shared_down"))


def out_errors(gpu: np.ndarray, ref: np.ndarray):
    diff = gpu.astype(np.float64) - ref
    rel = float(np.linalg.norm(diff) / max(np.linalg.norm(ref), 1e-30))
    return rel, float(np.abs(diff).max())


def check_routing(rec: dict, ref: dict, k: np.ndarray, E: int):
    """Bit-exact comparison of the integer routing record; alpha within
    ALPHA_RTOL (fp32 on the GPU, fp64 in the oracle)."""
    T, km = ref["ids"].shape
    assert np.array_equal(rec["ids"], ref["ids"]), "selected experts differ"
    valid = ref["ids"] >= 0
    np.testing.assert_allclose(rec["alpha"][valid], ref["alpha"][valid],
                               rtol=ALPHA_RTOL, atol=1e-7)
    assert np.all(rec["alpha"][~valid] == 0)
    assert np.array_equal(rec["offsets"], ref["offsets"]), "offsets differ"
    assert np.array_equal(rec["perm"], ref["perm"]), "permutation differs"
    assert np.array_equal(rec["row_of"], ref["row_of"]), "row_of differs"
    assert int(rec["totals"][0]) == int(k.sum()) == ref["perm"].size
    counts = np.diff(ref["offsets"])
    assert np.array_equal(rec["counts"], counts)
    assert int(rec["totals"][1]) == int(((counts + 127) // 128).sum())


def check_sampled_routing(rec: dict, layer: dict, k: np.ndarray, k_max: int,
                          tokens: np.ndarray, renorm: bool = True):
    """Routing of the listed tokens against the oracle run on those tokens
    only (scores are per token), plus properties of the whole record."""
    z = oracle.router_logits(layer["hidden"][tokens], layer["w_router"])
    ids, alpha = oracle.select(z, k[tokens], k_max, renorm)
    assert np.array_equal(rec["ids"][tokens], ids), "selected experts differ"
    valid = ids >= 0
    np.testing.assert_allclose(rec["alpha"][tokens][valid], alpha[valid],
                               rtol=ALPHA_RTOL, atol=1e-7)
    # whole record: pairs = sum k; perm is a permutation of the used slots
    # and row_of is its inverse; rows are grouped by expert in token order
    T = k.size
    n = int(k.sum())
    assert int(rec["totals"][0]) == n and rec["offsets"][-1] == n
    perm = rec["perm"]
    assert perm.size == n
    used = (np.arange(k_max)[None, :] < k[:, None]).ravel()
    assert np.array_equal(np.sort(perm), np.nonzero(used)[0])
    row_of = rec["row_of"].ravel()
    assert np.array_equal(row_of[perm], np.arange(n))
    assert np.all(row_of[~used] == -1)
    ids_all = rec["ids"].ravel()
    for e in range(len(rec["offsets"]) - 1):
        rows = perm[rec["offsets"][e]:rec["offsets"][e + 1]]
        assert np.all(ids_all[rows] == e)
        assert np.all(np.diff(rows) > 0)
