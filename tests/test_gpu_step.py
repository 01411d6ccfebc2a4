"""reflex_step (counts + forward in one call, the count kernel running beside
the router scores) against the two-call path reflex_allocate ->
reflex_moe_forward: every output bit for bit, on every layer shape, with the
App. C allocation variants, stage subsets, an allocation error, zero tokens
and CUDA-graph replay; plus the oracle on the LLaDA-MoE layer."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_01784_gb300 import _binding as B
from paper_2608_01784_gb300 import api
from paper_2608_01784_gb300 import workloads as W
from tests import gpu_cases as G

pytestmark = pytest.mark.gpu

RECORD = ("ids", "alpha", "counts", "offsets", "perm", "row_of", "totals", "scores")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_01784_gb300 import build
    build.build()
    B.load()
    oracle.build()


def _setup(name, seed):
    cfg = W.CONFIGS[name]
    layer = W.make_layer(cfg, seed)
    dl = api.layer_to_device(layer, cfg.dtype)
    moe = api.MoELayer(dl, dtype=cfg.dtype, d=cfg.d, E=cfg.E, inter=cfg.inter,
                       shared_inter=cfg.shared_inter, k_max=cfg.k_max, max_tokens=cfg.T)
    return cfg, layer, dl, moe


def _two_calls(moe, ds, p, hidden, flags):
    k, k_sum, st = api.allocate(ds, p)
    out = moe.forward(hidden, k, flags=flags)
    torch.cuda.synchronize()
    return out.clone(), k.clone(), k_sum.clone(), st.clone(), _record(moe)


def _one_call(moe, ds, p, hidden, flags):
    out, k, k_sum, st = moe.step(ds, p, hidden, flags=flags)
    torch.cuda.synchronize()
    return out.clone(), k.clone(), k_sum.clone(), st.clone(), _record(moe)


def _record(moe):
    return {k: v.clone() for k, v in moe.record().items()}


def _same(a, b, stages_run=True):
    out_a, k_a, s_a, st_a, rec_a = a
    out_b, k_b, s_b, st_b, rec_b = b
    assert torch.equal(k_a, k_b)
    assert torch.equal(s_a, s_b)
    assert B.reflex_read_status(st_a) == B.reflex_read_status(st_b)
    if stages_run:
        assert torch.equal(out_a.view(torch.int16) if out_a.dtype == torch.bfloat16 else out_a,
                           out_b.view(torch.int16) if out_b.dtype == torch.bfloat16 else out_b)
    for key in RECORD:
        assert torch.equal(rec_a[key], rec_b[key]), key


@pytest.mark.parametrize("name", ["tiny_fp32", "llada_moe", "llada2_mini", "llada_moe_b32"])
@pytest.mark.parametrize("variant", ["reflex", "fixed", "progress_only", "reflex_shuffled"])
def test_step_equals_allocate_then_forward(name, variant):
    from tests.test_gpu_parity import ALLOC_VARIANTS
    cfg, layer, dl, moe = _setup(name, 3)
    p = G.params_of(cfg, **ALLOC_VARIANTS[variant])
    for seed in range(2):
        ds = api.state_to_device(W.make_state(cfg, seed, hist_len=None))
        ref = _two_calls(moe, ds, p, dl["hidden"], B.REFLEX_FLAG_RENORM_TOPK)
        got = _one_call(moe, ds, p, dl["hidden"], B.REFLEX_FLAG_RENORM_TOPK)
        _same(ref, got)
        assert B.reflex_read_status(got[3]) == B.REFLEX_OK
        assert moe.status() == B.REFLEX_OK


@pytest.mark.parametrize("stages", [
    B.REFLEX_STAGE_ROUTE,
    B.REFLEX_STAGE_ROUTE | B.REFLEX_STAGE_DISPATCH,
    B.REFLEX_STAGE_DISPATCH,
])
def test_step_stage_subsets(stages):
    cfg, layer, dl, moe = _setup("llada2_mini", 5)
    p = G.params_of(cfg)
    ds = api.state_to_device(W.make_state(cfg, 1, hist_len=None))
    flags = B.REFLEX_FLAG_RENORM_TOPK | stages
    # the first full step fills the workspace, so stage subsets that skip
    # routing read the same routing on both paths
    moe.step(ds, p, dl["hidden"])
    ref = _two_calls(moe, ds, p, dl["hidden"], flags)
    got = _one_call(moe, ds, p, dl["hidden"], flags)
    _same(ref, got, stages_run=False)


def test_step_reports_allocation_errors_like_allocate():
    cfg, layer, dl, moe = _setup("llada2_mini", 7)
    p = G.params_of(cfg)
    state = W.make_state(cfg, 2, hist_len=None)
    state["active_block"][3] = 0          # no active block: flagged, counts kept valid
    ds = api.state_to_device(state)
    ref = _two_calls(moe, ds, p, dl["hidden"], B.REFLEX_FLAG_RENORM_TOPK)
    got = _one_call(moe, ds, p, dl["hidden"], B.REFLEX_FLAG_RENORM_TOPK)
    _same(ref, got)
    assert B.reflex_read_status(got[3]) != B.REFLEX_OK


def test_step_zero_tokens():
    cfg, layer, dl, moe = _setup("llada_moe", 1)
    p = G.params_of(cfg)
    ds = {k: v for k, v in api.state_to_device(W.make_state(cfg, 0)).items()}
    ds = dict(ds, conf1=ds["conf1"][:0], conf2=ds["conf2"][:0], hist_len=ds["hist_len"][:0],
              masked=ds["masked"][:0], block_id=ds["block_id"][:0],
              seq_offsets=torch.zeros(2, dtype=torch.int32, device="cuda"),
              active_block=torch.ones(1, dtype=torch.int32, device="cuda"))
    k_sum = torch.full((1,), 7, dtype=torch.int64, device="cuda")
    out, k, k_sum, st = moe.step(ds, p, dl["hidden"][:0], k_sum=k_sum)
    torch.cuda.synchronize()
    assert int(k_sum.item()) == 0 and B.reflex_read_status(st) == B.REFLEX_OK


def test_forward_zero_tokens_clears_a_stale_error():
    cfg, layer, dl, moe = _setup("llada_moe", 1)
    k = torch.full((cfg.T,), cfg.k_max + 3, dtype=torch.int32, device="cuda")
    moe.forward(dl["hidden"], k)                 # counts out of range: flagged
    torch.cuda.synchronize()
    assert moe.status() == B.REFLEX_EKRANGE
    moe.forward(dl["hidden"][:0], k[:0])
    torch.cuda.synchronize()
    assert moe.status() == B.REFLEX_OK


def test_step_graph_replay():
    cfg, layer, dl, moe = _setup("llada_moe", 2)
    p = G.params_of(cfg)
    ds = api.state_to_device(W.make_state(cfg, 4, hist_len=None))
    T = cfg.T
    out = torch.empty((T, cfg.d), dtype=torch.bfloat16, device="cuda")
    k = torch.empty(T, dtype=torch.int32, device="cuda")
    k_sum = torch.zeros(1, dtype=torch.int64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ref = _two_calls(moe, ds, p, dl["hidden"], B.REFLEX_FLAG_RENORM_TOPK)
    moe.step(ds, p, dl["hidden"], out=out, k_out=k, k_sum=k_sum, status=st)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="relaxed"):
        moe.step(ds, p, dl["hidden"], out=out, k_out=k, k_sum=k_sum, status=st)
    out.zero_()
    k.zero_()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    _same(ref, (out, k, k_sum, st, _record(moe)))


def test_step_llada_moe_against_oracle():
    cfg, layer, dl, moe = _setup("llada_moe", 0)
    state = W.make_state(cfg, 0)
    p = G.params_of(cfg)
    out, k, k_sum, st = moe.step(api.state_to_device(state), p, dl["hidden"])
    torch.cuda.synchronize()
    k_ref = G.oracle_allocate(state, p)
    assert np.array_equal(k.cpu().numpy(), k_ref)
    assert int(k_sum.item()) == int(k_ref.sum())
    ref = G.oracle_layer(cfg, layer, k_ref)
    G.check_routing({kk: v.cpu().numpy() for kk, v in moe.record().items()}, ref, k_ref, cfg.E)
    rel, mx = G.out_errors(G.to_f32(out), ref["out"])
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)


@pytest.mark.parametrize("name", ["llada_moe", "llada2_mini", "llada_moe_b32"])
def test_step_launch_count_matches_a_profile(name):
    # the bench's launch claim (api.step_launches) against the kernels a
    # profiler sees in one step; memsets are not kernels
    profiler = pytest.importorskip("torch.profiler")
    cfg, layer, dl, moe = _setup(name, 1)
    p = G.params_of(cfg)
    ds = api.state_to_device(W.make_state(cfg, 0, hist_len=None))
    moe.step(ds, p, dl["hidden"])          # warm: first-call attribute setup
    torch.cuda.synchronize()
    with profiler.profile(activities=[profiler.ProfilerActivity.CUDA]):
        moe.step(ds, p, dl["hidden"])      # warm the profiler itself
        torch.cuda.synchronize()
    with profiler.profile(activities=[profiler.ProfilerActivity.CUDA]) as prof:
        moe.step(ds, p, dl["hidden"])
        torch.cuda.synchronize()
    names = [e.name for e in prof.events()
             if e.device_type == torch.autograd.DeviceType.CUDA and "rx::" in e.name]
    if not names:
        pytest.skip("no kernel activity recorded by the profiler")
    assert len(names) == api.step_launches(cfg.dtype, cfg.T, cfg.d, cfg.E, cfg.shared_inter)
