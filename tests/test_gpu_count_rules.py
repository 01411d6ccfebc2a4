"""GPU parity of the score-based count rules (the threshold-based comparison
methods of App. B: Top-p and Expert-Threshold routing) on the same kernels as
REFLEX: the counts derived inside the TopK selection (reflex_step) and from a
score matrix (reflex_allocate) must equal the oracle's bit for bit, and the
layer run with them must match the oracle's layer (routing bit for bit,
outputs within the bf16 tolerance).  Thresholds are the paper's low / high
settings per model family (App. B), with the count bounds [1, 12]."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_01784_gb300 import _binding as B
from paper_2608_01784_gb300 import api
from paper_2608_01784_gb300 import workloads as W
from tests import gpu_cases as G

pytestmark = pytest.mark.gpu

TOP_P, THR = B.REFLEX_RULE_TOP_P, B.REFLEX_RULE_EXPERT_THRESHOLD
# (p of Top-p; expert threshold) low / high, App. B
LLADA_MOE = [(TOP_P, 0.15), (TOP_P, 0.20), (THR, 0.0215), (THR, 0.0190)]
LLADA2_MINI = [(TOP_P, 0.25), (TOP_P, 0.325), (THR, 0.0270), (THR, 0.0220)]


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_01784_gb300 import build
    build.build()
    B.load()
    oracle.build()


def _rule_params(cfg, rule, thr, k_min=1, k_max=12):
    return G.params_of(cfg, count_rule=rule, rule_threshold=thr, k_min=k_min,
                       k_max=min(k_max, cfg.k_max))


def _step(cfg, layer, state, p, flags=B.REFLEX_FLAG_RENORM_TOPK):
    gl = G.GpuLayer(cfg, layer)
    ds = api.state_to_device(state)
    out, k, ks, st = gl.moe.step(ds, p, gl.dev["hidden"], flags=flags)
    torch.cuda.synchronize()
    assert B.reflex_read_status(st) == B.REFLEX_OK
    assert gl.moe.status() == B.REFLEX_OK
    rec = {n: v.cpu().numpy() for n, v in gl.moe.record().items()}
    return G.to_f32(out), k.cpu().numpy(), int(ks.item()), rec


@pytest.mark.parametrize("rule,thr", LLADA_MOE)
def test_step_rule_counts_llada_moe_layer(rule, thr):
    cfg = W.CONFIGS["llada_moe"]
    layer, state = W.make_layer(cfg, 21), W.make_state(cfg, 21)
    p = _rule_params(cfg, rule, thr)
    out, k, ks, rec = _step(cfg, layer, state, p)
    z = oracle.router_logits(layer["hidden"], layer["w_router"])
    k_ref = oracle.rule_counts(z, rule, thr, 1, 12)
    assert np.array_equal(k, k_ref)
    assert ks == int(k_ref.sum())
    assert 1 < k_ref.mean() < 12            # the threshold decides something
    ref = G.oracle_layer(cfg, layer, k_ref)
    G.check_routing(rec, ref, k_ref, cfg.E)
    rel, mx = G.out_errors(out, ref["out"])
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)


@pytest.mark.parametrize("rule,thr", LLADA2_MINI)
def test_step_rule_counts_llada2_mini_layer(rule, thr):
    # 256 experts: the score rules read every score, so this forward scores
    # every expert with the chain (no screen); outputs on sampled tokens
    cfg = W.CONFIGS["llada2_mini"]
    layer, state = W.make_layer(cfg, 22), W.make_state(cfg, 22)
    p = _rule_params(cfg, rule, thr)
    out, k, ks, rec = _step(cfg, layer, state, p)
    z = oracle.router_logits(layer["hidden"], layer["w_router"])
    k_ref = oracle.rule_counts(z, rule, thr, 1, 12)
    assert np.array_equal(k, k_ref)
    assert ks == int(k_ref.sum())
    ids, alpha = oracle.select(z, k_ref, cfg.k_max)
    offsets, perm, row_of = oracle.permutation(ids, k_ref, cfg.E)
    ref = dict(ids=ids, alpha=alpha, offsets=offsets, perm=perm, row_of=row_of)
    G.check_routing(rec, ref, k_ref, cfg.E)
    toks = W.sample_tokens(state, stride=131)
    want = oracle.moe_tokens(layer["hidden"], layer["w_gate_up"], layer["w_down"], ids,
                             alpha, k_ref, toks, shared_gate_up=layer["shared_gate_up"],
                             shared_down=layer["shared_down"])
    rel, mx = G.out_errors(out[toks], want)
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)


def test_step_rule_counts_tiny_fp32_and_the_clip():
    cfg = W.CONFIGS["tiny_fp32"]
    layer, state = W.make_layer(cfg, 23), W.make_state(cfg, 23)
    z = oracle.router_logits(layer["hidden"], layer["w_router"])
    for rule, thr, lo in ((TOP_P, 0.5, 1), (TOP_P, 0.99, 2), (THR, 0.1, 1), (THR, 0.3, 2)):
        p = _rule_params(cfg, rule, thr, k_min=lo, k_max=4)
        out, k, ks, rec = _step(cfg, layer, state, p)
        k_ref = oracle.rule_counts(z, rule, thr, lo, 4)
        assert np.array_equal(k, k_ref), (rule, thr)
        ref = G.oracle_layer(cfg, layer, k_ref)
        G.check_routing(rec, ref, k_ref, cfg.E)
        rel, mx = G.out_errors(out, ref["out"])
        assert rel <= G.F32_REL_L2 and mx <= G.F32_MAX_ABS, (rel, mx)


@pytest.mark.parametrize("E", [8, 64, 256, 1000])
def test_allocate_from_router_scores(E):
    # reflex_allocate with a score matrix: counts only, any E up to 1024
    # (ragged lane groups at E = 1000); scores span several scales, and
    # exact ties and equal rows are included
    rng = np.random.default_rng(E)
    T = 3000
    z = (rng.standard_normal((T, E)) * rng.uniform(0.05, 4.0, (T, 1))).astype(np.float32)
    z[5] = 0.25                                   # every expert equal
    z[6, : E // 2] = z[6, E // 2: 2 * (E // 2)]   # pairs of equal scores
    zd = torch.from_numpy(z).cuda()
    cfg = W.CONFIGS["llada_moe"]
    for rule, thr in ((TOP_P, 0.2), (TOP_P, 0.6), (THR, 1.5 / E), (THR, 0.02)):
        p = _rule_params(cfg, rule, thr)
        k, ks, st = api.allocate(None, p, router_scores=zd)
        torch.cuda.synchronize()
        assert B.reflex_read_status(st) == B.REFLEX_OK
        k_ref = oracle.rule_counts(z, rule, thr, 1, 12)
        assert np.array_equal(k.cpu().numpy(), k_ref), (rule, thr)
        assert int(ks.item()) == int(k_ref.sum())


def test_step_rule_graph_replay_and_fixed_state():
    # the counts follow the router, not the refinement state: a different
    # state gives the same counts; a captured step replays to the same bits
    cfg = W.CONFIGS["llada_moe"]
    layer = W.make_layer(cfg, 24)
    p = _rule_params(cfg, TOP_P, 0.2)
    out_a, k_a, _, _ = _step(cfg, layer, W.make_state(cfg, 1), p)
    out_b, k_b, _, _ = _step(cfg, layer, W.make_state(cfg, 2), p)
    assert np.array_equal(k_a, k_b) and np.array_equal(out_a, out_b)
    gl = G.GpuLayer(cfg, layer)
    ds = api.state_to_device(W.make_state(cfg, 3))
    out = torch.empty_like(gl.dev["hidden"])
    k = torch.empty(cfg.T, dtype=torch.int32, device="cuda")
    ks = torch.zeros(1, dtype=torch.int64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="relaxed"):
        gl.moe.step(ds, p, gl.dev["hidden"], out=out, k_out=k, k_sum=ks, status=st)
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    assert np.array_equal(G.to_f32(out), out_a)
    assert np.array_equal(k.cpu().numpy(), k_a) and int(ks.item()) == int(k_a.sum())
