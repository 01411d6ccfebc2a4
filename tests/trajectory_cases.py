"""Trajectory drivers shared by the CPU pins and the GPU parity tests: the
oracle's trajectory (oracle allocation and state update on host arrays) with
the same synthetic confidences the device driver uses (computed on CPU
tensors; the model is exact fp32 arithmetic, so CPU and CUDA agree)."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2608_01784_gb300 import trajectory as TR


def oracle_trajectory(state: dict, params: dict, seed: int = 0, theta: float = 0.9,
                      max_forwards: int = 100000):
    """Returns (per-forward counts, NFE per sequence, pairs per sequence,
    final state) of the oracle's run from `state` (numpy, not modified)."""
    st = {k: np.array(v, copy=True) for k, v in state.items()}
    nb = TR.num_blocks(st)
    sidx_np = TR.seq_index(st)
    sidx = torch.from_numpy(sidx_np)
    B = nb.size
    nfe = np.zeros(B, np.int64)
    pairs = np.zeros(B, np.int64)
    ks = []
    for t in range(max_forwards):
        running = st["active_block"] <= nb
        if not running.any():
            break
        k = oracle.allocate(st["conf1"], st["conf2"], st["hist_len"], st["masked"],
                            st["block_id"], st["seq_offsets"], st["active_block"], **params)
        ks.append(k)
        nfe += running
        pairs += np.bincount(sidx_np, weights=k, minlength=B).astype(np.int64) * running
        conf = TR.synthetic_confidence({kk: torch.from_numpy(np.asarray(v)) for kk, v in st.items()},
                                       t, seed, sidx).numpy()
        st, _ = oracle.update_state(st, conf, nb, theta)
    return ks, nfe, pairs, st
