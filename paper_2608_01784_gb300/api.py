"""Torch-facing convenience over the C ABI: device buffers, workspace and
route-record views.  PyTorch provides memory and streams only; every step of
the path runs in libreflex.so's kernels.
"""
from __future__ import annotations

import numpy as np
import torch

from . import _binding as B


def _dev(a: np.ndarray, device, dtype=None) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.view(dtype)
    return t.to(device, non_blocking=False)


def layer_to_device(layer: dict, dtype: str, device="cuda") -> dict:
    """Host arrays (fp32, or bf16 bit patterns as uint16) -> device tensors."""
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    out = {}
    for k, v in layer.items():
        if v.dtype == np.uint16:
            out[k] = _dev(v.view(np.int16), device).view(tdt)
        else:
            out[k] = _dev(v, device)
    return out


def state_to_device(state: dict, device="cuda") -> dict:
    return {k: _dev(v, device) for k, v in state.items()}


def allocate(state: dict, params: B.reflex_alloc_params, E: int = 0,
             stream=None, k_out: torch.Tensor | None = None,
             k_sum: torch.Tensor | None = None,
             status: torch.Tensor | None = None,
             router_scores: torch.Tensor | None = None):
    """reflex_allocate on device state tensors -> (k int32 [T], k_sum int64 [1],
    status int32 [1]).  With a score rule (params.count_rule) the counts come
    from router_scores [T, E] fp32 and `state` may be None."""
    if router_scores is not None:
        T, E = int(router_scores.shape[0]), int(router_scores.shape[1])
        dev = router_scores.device
        nseq = 1
    else:
        T = int(state["block_id"].numel())
        nseq = int(state["active_block"].numel())
        dev = state["block_id"].device
    k_out = torch.empty(T, dtype=torch.int32, device=dev) if k_out is None else k_out
    k_sum = torch.zeros(1, dtype=torch.int64, device=dev) if k_sum is None else k_sum
    status = torch.zeros(1, dtype=torch.int32, device=dev) if status is None else status
    st = state if state is not None else {}
    B.reflex_allocate(router_scores, st.get("conf1"), st.get("conf2"), st.get("hist_len"),
                      st.get("masked"), st.get("block_id"), st.get("seq_offsets"),
                      st.get("active_block"), T, nseq, E, params, k_out, k_sum,
                      status, stream)
    return k_out, k_sum, status


def update_state(state: dict, conf_new: torch.Tensor, num_blocks: torch.Tensor,
                 theta_commit: float, stream=None,
                 committed: torch.Tensor | None = None,
                 status: torch.Tensor | None = None):
    """reflex_update_state in place on device state tensors (Eq. 1 commits,
    confidence history, active-block advance); returns committed [B]."""
    T = int(state["block_id"].numel())
    nseq = int(state["active_block"].numel())
    dev = state["block_id"].device
    committed = (torch.empty(nseq, dtype=torch.int32, device=dev)
                 if committed is None else committed)
    B.reflex_update_state(conf_new, state["conf1"], state["conf2"], state["hist_len"],
                          state["masked"], state["block_id"], state["seq_offsets"],
                          state["active_block"], num_blocks, T, nseq, theta_commit,
                          committed, status, stream)
    return committed


def step_launches(dtype: str, T: int, d: int, E: int, shared_inter: int,
                  flags: int = B.REFLEX_FLAG_RENORM_TOPK, count_rule: int = 0) -> int:
    """Kernels one reflex_step call launches on the tcgen05 path, following the
    library's choices: the count kernel; the score kernel and the selection,
    or (bf16, renormalised weights, >= 128 experts, T E >= 2048 x 256,
    d % 128 == 0) the norm kernel, the score GEMM and the screened selection,
    or (bf16, renormalised weights, at most 64 experts and >= 8192 tokens, or
    65-256 experts and >= 2048 tokens) the norm kernel, the score GEMM and
    the batched recheck; count + scan in one
    CTA (short batches whose block masks fit in shared memory) or count and
    scan, then the gather, which also places the pairs; the gate/up and down
    GEMMs (and the shared expert's two); the combine.
    With a score count rule the selection derives the counts: no count
    kernel and no screen.  Memsets are not kernels."""
    n = 0 if count_rule else 1
    screened = (dtype == "bf16" and flags & B.REFLEX_FLAG_RENORM_TOPK and
                not flags & B.REFLEX_FLAG_EXACT_SCORES and not count_rule)
    screen = screened and d % 128 == 0 and E >= 128 and T * E >= 2048 * 256
    batch_screen = screened and d % 64 == 0 and (
        (E <= 64 and T >= 8192) or (64 < E <= 256 and T >= 2048))
    n += 3 if (screen or batch_screen) else 2
    n += 1 if T <= 4096 and (T + 31) // 32 * E * 4 <= 160 * 1024 else 2
    n += 1 + 2 + (2 if shared_inter else 0) + 1
    return n


class MoELayer:
    """One variable-count MoE layer on the device with its workspace sized for
    `max_tokens` tokens at `k_max`."""

    def __init__(self, weights: dict, *, dtype: str, d: int, E: int, inter: int,
                 shared_inter: int, k_max: int, max_tokens: int, device="cuda"):
        self.w = weights
        self.dtype = B.REFLEX_DTYPE_BF16 if dtype == "bf16" else B.REFLEX_DTYPE_F32
        self.tdtype = torch.bfloat16 if dtype == "bf16" else torch.float32
        self.d, self.E, self.inter = d, E, inter
        self.shared_inter = shared_inter
        self.k_max = k_max
        self.max_tokens = max_tokens
        self.ws_bytes = B.reflex_moe_workspace_size(self.dtype, max_tokens, d, E,
                                                    inter, shared_inter, k_max)
        if self.ws_bytes == 0:
            raise ValueError("unsupported MoE layer shape")
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=device)
        self.rec = B.reflex_route_record()
        self._T = 0

    def forward(self, hidden: torch.Tensor, k: torch.Tensor, out=None,
                flags: int = B.REFLEX_FLAG_RENORM_TOPK, stream=None,
                check: bool = True) -> torch.Tensor:
        T = int(hidden.shape[0])
        if T > self.max_tokens:
            raise ValueError("more tokens than the workspace was sized for")
        if out is None:
            out = torch.empty((T, self.d), dtype=self.tdtype, device=hidden.device)
        B.reflex_moe_forward(self.dtype, hidden, self.w["w_router"],
                             self.w["w_gate_up"], self.w["w_down"],
                             self.w.get("shared_gate_up"), self.w.get("shared_down"),
                             self.shared_inter, k, T, self.d, self.E, self.inter,
                             self.k_max, flags, self.ws, self.ws_bytes, out, self.rec,
                             stream, check)
        self._T = T
        return out

    def step(self, state: dict, params: B.reflex_alloc_params, hidden: torch.Tensor,
             out=None, k_out: torch.Tensor | None = None,
             k_sum: torch.Tensor | None = None, status: torch.Tensor | None = None,
             flags: int = B.REFLEX_FLAG_RENORM_TOPK, stream=None, check: bool = True):
        """reflex_step: the counts of `state` (as allocate) and the forward with
        them in one call -> (out, k int32 [T], k_sum int64 [1], status int32 [1])."""
        T = int(hidden.shape[0])
        if T > self.max_tokens:
            raise ValueError("more tokens than the workspace was sized for")
        if int(state["block_id"].numel()) != T:
            raise ValueError("state and hidden disagree on the token count")
        dev = hidden.device
        nseq = int(state["active_block"].numel())
        out = torch.empty((T, self.d), dtype=self.tdtype, device=dev) if out is None else out
        k_out = torch.empty(T, dtype=torch.int32, device=dev) if k_out is None else k_out
        k_sum = torch.zeros(1, dtype=torch.int64, device=dev) if k_sum is None else k_sum
        status = torch.zeros(1, dtype=torch.int32, device=dev) if status is None else status
        B.reflex_step(state["conf1"], state["conf2"], state["hist_len"], state["masked"],
                      state["block_id"], state["seq_offsets"], state["active_block"],
                      nseq, params, k_out, k_sum, status, self.dtype, hidden,
                      self.w["w_router"], self.w["w_gate_up"], self.w["w_down"],
                      self.w.get("shared_gate_up"), self.w.get("shared_down"),
                      self.shared_inter, T, self.d, self.E, self.inter, self.k_max,
                      flags, self.ws, self.ws_bytes, out, self.rec, stream, check)
        self._T = T
        return out, k_out, k_sum, status

    def status(self, stream=None) -> int:
        return B.reflex_moe_status(self.ws, stream)

    def _view(self, addr: int, n: int, dtype=torch.int32) -> torch.Tensor:
        off = addr - self.ws.data_ptr()
        nbytes = n * torch.empty((), dtype=dtype).element_size()
        return self.ws[off:off + nbytes].view(dtype)

    def record(self) -> dict:
        """Views (no copies) of the routing record of the last forward."""
        T, km, E = self._T, self.k_max, self.E
        totals = self._view(self.rec.totals, 2)
        n_pairs = int(totals[0].item())
        return dict(
            ids=self._view(self.rec.ids, T * km).view(T, km),
            alpha=self._view(self.rec.alpha, T * km, torch.float32).view(T, km),
            counts=self._view(self.rec.counts, E),
            offsets=self._view(self.rec.offsets, E + 1),
            perm=self._view(self.rec.perm, n_pairs),
            row_of=self._view(self.rec.row_of, T * km).view(T, km),
            totals=totals,
            scores=self._view(self.rec.scores, T * E, torch.float32).view(T, E),
        )


class MoEStack:
    """A stack of variable-count MoE layers of one shape sharing one workspace:
    one denoising forward computes the per-token counts once (Eq. 3; the
    counts are shared by every layer) and runs every layer with the residual
    connection h <- h + MoE(h).  The first layer runs with the counts in one
    reflex_step call, the others with reflex_moe_forward; every call takes the
    current stream, so a whole forward can be captured in one CUDA graph."""

    def __init__(self, layers: list, *, dtype: str, d: int, E: int, inter: int,
                 shared_inter: int, k_max: int, max_tokens: int, device="cuda"):
        if not layers:
            raise ValueError("a stack needs at least one layer")
        self.layers = layers
        self.moe = MoELayer(layers[0], dtype=dtype, d=d, E=E, inter=inter,
                            shared_inter=shared_inter, k_max=k_max,
                            max_tokens=max_tokens, device=device)
        self.d, self.E = d, E
        self.tdtype = self.moe.tdtype
        self._bufs = [torch.empty((max_tokens, d), dtype=self.tdtype, device=device)
                      for _ in range(2)]

    def _layer_out(self, l: int, T: int, out: torch.Tensor, keep):
        if keep is not None:
            return keep[l]
        if l == len(self.layers) - 1:
            return out
        return self._bufs[l & 1][:T]

    def forward(self, state: dict, params: B.reflex_alloc_params, hidden: torch.Tensor,
                out: torch.Tensor, k_out: torch.Tensor, k_sum: torch.Tensor,
                status: torch.Tensor, flags: int = B.REFLEX_FLAG_RENORM_TOPK,
                keep: list | None = None, around_up=None, check: bool = True):
        """One denoising forward: `out` receives the last layer's output.
        `keep` (optional) lists one [T, d] tensor per layer that receives that
        layer's output instead of the internal ping-pong buffers.
        `around_up` (optional) is a pair of callables run right before and
        after every layer's gate/up GEMM (the layer is then issued as three
        stage calls on the same workspace, which gives the same bits)."""
        T = int(hidden.shape[0])
        flags = flags | B.REFLEX_FLAG_RESIDUAL
        h = hidden
        for l, w in enumerate(self.layers):
            self.moe.w = w
            dst = self._layer_out(l, T, out, keep)
            if around_up is None:
                if l == 0:
                    self.moe.step(state, params, h, out=dst, k_out=k_out, k_sum=k_sum,
                                  status=status, flags=flags, check=check)
                else:
                    self.moe.forward(h, k_out, dst, flags, check=check)
            else:
                first = B.REFLEX_STAGE_ROUTE | B.REFLEX_STAGE_DISPATCH
                if l == 0:
                    self.moe.step(state, params, h, out=dst, k_out=k_out, k_sum=k_sum,
                                  status=status, flags=flags | first, check=check)
                else:
                    self.moe.forward(h, k_out, dst, flags | first, check=check)
                around_up[0](l)
                self.moe.forward(h, k_out, dst, flags | B.REFLEX_STAGE_EXPERT_UP,
                                 check=check)
                around_up[1](l)
                self.moe.forward(h, k_out, dst, flags | B.REFLEX_STAGE_EXPERT_DOWN |
                                 B.REFLEX_STAGE_COMBINE, check=check)
            h = dst
        return out

    def status(self) -> int:
        return self.moe.status()
