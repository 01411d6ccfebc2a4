"""Denoising-trajectory driver: repeats allocation -> MoE layer -> state update
over the forwards of block-wise inference until every sequence has resolved
its blocks (Sec. 3.1), and reports forwards (NFE) and selected expert-token
pairs per sequence (the paper's computation metric, Sec. 3.2).

There is no language model here.  The confidences a forward would produce
come from a synthetic model (`synthetic_confidence`): a masked position's
confidence rises by a block-distance-dependent gain plus seeded noise each
forward.  It is built from exact fp32 operations (+, -, x, clamp) and a 31-bit
integer hash, so CPU and CUDA tensors give identical values; that lets tests
run the GPU trajectory and the oracle trajectory side by side.
"""
from __future__ import annotations

import numpy as np
import torch

from . import _binding as B
from . import api

# gain per forward by distance to the active block, noise amplitude, initial
# confidence range of a never-predicted position
GAIN_ACTIVE = 0.09
GAIN_NEXT = 0.03
GAIN_FAR = 0.01
NOISE = 0.12
INIT_LO = 0.05
INIT_SPAN = 0.25


def num_blocks(state: dict) -> np.ndarray:
    """Q of every sequence: its largest block id."""
    bid = np.asarray(state["block_id"])
    so = np.asarray(state["seq_offsets"])
    return np.array([int(bid[so[s]:so[s + 1]].max(initial=0)) for s in range(so.size - 1)],
                    np.int32)


def initial_state(state: dict) -> dict:
    """The start of generation for the layout of `state` (numpy): every
    target position masked, block 1 active, no confidence observed yet."""
    st = {k: np.array(v, copy=True) for k, v in state.items()}
    st["masked"] = (np.asarray(st["block_id"]) > 0).astype(np.uint8)
    st["active_block"] = np.ones_like(np.asarray(st["active_block"]), dtype=np.int32)
    st["hist_len"] = np.zeros_like(np.asarray(st["hist_len"]), dtype=np.uint8)
    st["conf1"] = np.zeros_like(np.asarray(st["conf1"]), dtype=np.float32)
    st["conf2"] = np.zeros_like(np.asarray(st["conf2"]), dtype=np.float32)
    return st


def seq_index(state: dict) -> np.ndarray:
    so = np.asarray(state["seq_offsets"])
    return np.repeat(np.arange(so.size - 1), np.diff(so)).astype(np.int64)


def _uniform24(seed: int, t, idx: torch.Tensor) -> torch.Tensor:
    """Seeded uniform in [0, 1) with 24 bits per (seed, forward, position);
    every intermediate stays below 2^63 in int64.  t is an int or an int64
    tensor on idx's device (a graph-replayed loop keeps it on the device)."""
    m = 0x7FFFFFFF
    x = (idx * 2654435761 + (t * 1013904223 + (seed & m) * 362437)) & m
    x = x ^ (x >> 15)
    x = (x * 2246822519) & m
    x = x ^ (x >> 13)
    x = (x * 3266489917) & m
    x = x ^ (x >> 16)
    return (x >> 7).to(torch.float32) * (1.0 / 16777216.0)


def synthetic_confidence(state: dict, t, seed: int, seq_idx: torch.Tensor) -> torch.Tensor:
    """Confidences of forward t for every position (meaningful where masked):
    clamp(previous + gain(|b - a|) + NOISE (u - 1/2), 0, 1), previous = the
    last observation, or a seeded initial value for a position never
    predicted."""
    dev = state["block_id"].device
    idx = torch.arange(state["block_id"].numel(), dtype=torch.int64, device=dev)
    a = state["active_block"].to(torch.int64)[seq_idx]
    dist = (state["block_id"].to(torch.int64) - a).abs()
    gain = torch.where(dist == 0, GAIN_ACTIVE,
                       torch.where(dist == 1, GAIN_NEXT, GAIN_FAR)).to(torch.float32)
    init = _uniform24(seed, 0, idx) * INIT_SPAN + INIT_LO
    prev = torch.where(state["hist_len"] > 0, state["conf1"], init)
    noise = (_uniform24(seed, t + 1, idx) - 0.5) * NOISE
    return torch.clamp((prev + gain) + noise, 0.0, 1.0)


def simulate(state: dict, params: B.reflex_alloc_params, E: int, *, theta_commit: float = 0.9,
             seed: int = 0, max_forwards: int = 100000, moe: api.MoELayer | None = None,
             hidden: torch.Tensor | None = None, layers: int = 1, check_every: int = 1,
             record=None, graph: bool = False) -> dict:
    """Runs forwards on the device state (modified in place) until every
    sequence is finished.  With `moe` and `hidden`, each forward also runs
    `layers` MoE layers at the allocated counts (the cost of the forward; the
    synthetic confidences do not depend on their output).  With `graph`, one
    forward is captured as a CUDA graph and replayed (the forward index lives
    on the device), so the loop is not bound by host launches; finished
    sequences make later replays no-ops, and completion is checked every
    `check_every` forwards.  Returns per sequence NFE and pairs (per layer)
    and the number of forwards run."""
    dev = state["block_id"].device
    nb = torch.from_numpy(num_blocks({k: v.cpu() for k, v in state.items()})).to(dev)
    sidx = torch.from_numpy(seq_index({"seq_offsets": state["seq_offsets"].cpu()})).to(dev)
    Bn = int(state["active_block"].numel())
    T = int(state["block_id"].numel())
    k = torch.empty(T, dtype=torch.int32, device=dev)
    ksum = torch.zeros(1, dtype=torch.int64, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    upd_status = torch.zeros(1, dtype=torch.int32, device=dev)
    committed = torch.empty(Bn, dtype=torch.int32, device=dev)
    nfe = torch.zeros(Bn, dtype=torch.int64, device=dev)
    pairs = torch.zeros(Bn, dtype=torch.int64, device=dev)
    out = None
    if moe is not None:
        out = torch.empty((T, moe.d), dtype=moe.tdtype, device=dev)
    def forward(t):
        running = (state["active_block"] <= nb).to(torch.int64)
        if moe is not None:   # counts and the first layer in one call
            moe.step(state, params, hidden, out=out, k_out=k, k_sum=ksum, status=status)
            for _ in range(layers - 1):
                moe.forward(hidden, k, out)
        else:
            api.allocate(state, params, E, None, k, ksum, status)
        nfe.add_(running)
        pairs.add_(torch.zeros(Bn, dtype=torch.int64, device=dev).index_add_(
            0, sidx, k.to(torch.int64)) * running)
        conf = synthetic_confidence(state, t, seed, sidx)
        api.update_state(state, conf, nb, theta_commit, committed=committed, status=upd_status)

    def done() -> bool:
        return not bool((state["active_block"] <= nb).any())

    forwards = 0
    if graph:
        t_dev = torch.zeros((), dtype=torch.int64, device=dev)

        def body():
            forward(t_dev)
            t_dev.add_(1)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="relaxed"):
            body()
        while forwards < max_forwards:
            if forwards % check_every == 0 and done():
                break
            g.replay()
            forwards += 1
    else:
        for t in range(max_forwards):
            if t % check_every == 0 and done():
                break
            forward(t)
            if record is not None:
                record.append(k.clone())
            forwards += 1
    return dict(nfe=nfe.cpu().numpy(), pairs=pairs.cpu().numpy(), forwards=forwards,
                alloc_status=B.reflex_read_status(status),
                update_status=B.reflex_read_status(upd_status))
