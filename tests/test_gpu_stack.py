"""The 16-layer stack at full size (the bench's default workload): a whole
denoising forward through api.MoEStack (counts once, Eq. 3; every layer
Eq. 2 with the residual h <- bf16(h + MoE(h)); reading: layer chaining).

Parity is taken layer by layer on sampled tokens: the oracle runs layer l on
the GPU's own bf16 input of layer l, so routing stays comparable bit for bit
in every layer (a drift over 16 layers would say nothing about one layer).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_01784_gb300 import _binding as B
from paper_2608_01784_gb300 import api
from paper_2608_01784_gb300 import workloads as W
from tests import gpu_cases as G

pytestmark = pytest.mark.gpu

L = 16


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_01784_gb300 import build
    build.build()
    B.load()


@pytest.fixture(scope="module")
def stack_run():
    cfg = W.CONFIGS["llada_moe_b32"]
    seed = 5
    stack = W.make_stack(cfg, seed, L)
    state = W.make_state(cfg, seed)
    ds = api.state_to_device(state)
    layers = [api.layer_to_device(w, cfg.dtype) for w in stack["layers"]]
    h0 = api.layer_to_device({"hidden": stack["hidden"]}, cfg.dtype)["hidden"]
    net = api.MoEStack(layers, dtype=cfg.dtype, d=cfg.d, E=cfg.E, inter=cfg.inter,
                       shared_inter=0, k_max=cfg.k_max, max_tokens=cfg.T)
    T = cfg.T
    keep = [torch.empty_like(h0) for _ in range(L)]
    k = torch.empty(T, dtype=torch.int32, device="cuda")
    ks = torch.zeros(1, dtype=torch.int64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    p = G.params_of(cfg)
    net.forward(ds, p, h0, keep[-1], k, ks, st, keep=keep)
    torch.cuda.synchronize()
    assert B.reflex_read_status(st) == B.REFLEX_OK
    assert net.status() == B.REFLEX_OK
    rec = {n: v.cpu().numpy() for n, v in net.moe.record().items()}
    outs = [x.view(torch.int16).cpu().numpy().view(np.uint16) for x in keep]
    # the same forward as one CUDA-graph replay into the ping-pong buffers
    out = torch.empty_like(h0)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="relaxed"):
        net.forward(ds, p, h0, out, k, ks, st)
    g.replay()
    torch.cuda.synchronize()
    graph_out = out.view(torch.int16).cpu().numpy().view(np.uint16)
    rng = np.random.default_rng(seed)
    tokens = np.sort(rng.choice(T, 48, replace=False)).astype(np.int32)
    return dict(cfg=cfg, stack=stack, state=state, p=p, k=k.cpu().numpy(),
                k_sum=int(ks.item()), outs=outs, rec=rec, graph_out=graph_out,
                tokens=tokens)


def test_stack_counts_are_allocated_once_and_bit_exact(stack_run):
    r = stack_run
    k_ref = G.oracle_allocate(r["state"], r["p"])
    assert np.array_equal(r["k"], k_ref)
    assert r["k_sum"] == int(k_ref.sum())


def test_stack_graph_replay_gives_the_eager_bits(stack_run):
    assert np.array_equal(stack_run["graph_out"], stack_run["outs"][-1])


def test_stack_every_layer_on_sampled_tokens(stack_run):
    r = stack_run
    cfg, toks, k = r["cfg"], r["tokens"], r["k"]
    for l in range(L):
        h_in = r["stack"]["hidden"] if l == 0 else r["outs"][l - 1]
        w = r["stack"]["layers"][l]
        res = oracle.moe_layer(h_in[toks], w["w_router"], w["w_gate_up"], w["w_down"],
                               k[toks], cfg.k_max)
        ref_bits = oracle.residual_bf16(h_in[toks], res["out"])
        ref = W.bf16_bits_to_f32(ref_bits).astype(np.float64)
        gpu = W.bf16_bits_to_f32(r["outs"][l][toks])
        rel, mx = G.out_errors(gpu, ref)
        assert rel <= G.BF16_REL_L2, (l, rel)
        assert G.residual_excess(gpu, ref, rounded_ref=True) <= 0, (l, mx)
        if l == L - 1:   # the record holds the last layer's routing
            G.check_sampled_routing(r["rec"], dict(hidden=h_in, w_router=w["w_router"]),
                                    k, cfg.k_max, toks)
