"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the
same seeded inputs.  Allocation, selected experts, pair offsets and the pair
permutation must match bit for bit; router weights within 2e-5 relative;
layer outputs within rel-L2 1e-2 / max-abs 2e-2 for bf16 storage with fp32
accumulation (1e-5 / 1e-4 for fp32 storage)."""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2608_01784_gb300 import _binding as B
from paper_2608_01784_gb300 import api
from paper_2608_01784_gb300 import workloads as W
from tests import gpu_cases as G

pytestmark = pytest.mark.gpu

CFG = W.CONFIGS


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_01784_gb300 import build
    build.build()
    B.load()
    oracle.build()


# ---------------------------------------------------------------------------
# bounded waits
# ---------------------------------------------------------------------------
def test_wait_timeout_is_reported_and_context_survives():
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert B.reflex_selftest_wait_timeout(st, 2000) == B.REFLEX_OK
    assert B.reflex_read_status(st) == B.REFLEX_ETIMEOUT
    # the context is still usable afterwards
    cfg = CFG["tiny_fp32"]
    state = W.make_state(cfg, 0)
    k, ksum, status = G.gpu_allocate(state, G.params_of(cfg))
    assert status == B.REFLEX_OK and ksum == int(k.sum())


# ---------------------------------------------------------------------------
# allocation (Eq. 5, Eq. 6-9, clip)
# ---------------------------------------------------------------------------
ALLOC_VARIANTS = {
    "reflex": {},
    "fixed": dict(delta_role=0, delta_cur=0),
    "rrb_only": dict(delta_cur=0),
    "fger_only": dict(delta_role=0),
    "wide_clip": dict(k_max=14),
    "tight_tau": dict(tau=0.01),
    # App. C ablations: rank keys of the Eq. 9 groups, Role-Shuffled RRB
    "frontier_only": dict(signal=B.REFLEX_SIGNAL_FRONTIER),
    "progress_only": dict(signal=B.REFLEX_SIGNAL_PROGRESS),
    "confidence_only": dict(signal=B.REFLEX_SIGNAL_CONFIDENCE),
    "uncertainty_only": dict(signal=B.REFLEX_SIGNAL_UNCERTAINTY),
    "role_shuffled_rrb": dict(delta_cur=0, role_shuffle=1, shuffle_seed=12345),
    "reflex_shuffled": dict(role_shuffle=1, shuffle_seed=2**63 + 7),
}


@pytest.mark.parametrize("name", ["tiny_fp32", "llada_moe", "llada2_mini", "llada_moe_b32"])
@pytest.mark.parametrize("hist", [0, 1, 2])
@pytest.mark.parametrize("variant", list(ALLOC_VARIANTS))
def test_allocate_bit_exact(name, hist, variant):
    cfg = CFG[name]
    for seed in range(3):
        state = W.make_state(cfg, seed, hist_len=hist)
        p = G.params_of(cfg, **ALLOC_VARIANTS[variant])
        k_gpu, ksum, status = G.gpu_allocate(state, p)
        k_ref = G.oracle_allocate(state, p)
        assert status == B.REFLEX_OK
        assert np.array_equal(k_gpu, k_ref)
        assert ksum == int(k_ref.sum())


def test_allocate_role_shuffle_long_sequence_flags_capacity():
    # one 8192-token sequence: longer than the shuffle's 4096-token limit, so
    # the counts stay unshuffled and REFLEX_ECAPACITY is reported
    cfg = CFG["llada2_mini"]
    state = W.make_state(cfg, 3)
    state["seq_offsets"] = np.array([0, state["block_id"].size], np.int32)
    state["active_block"] = state["active_block"][:1].copy()
    p = G.params_of(cfg, delta_cur=0, role_shuffle=1, shuffle_seed=9)
    k_gpu, ksum, status = G.gpu_allocate(state, p)
    assert status == B.REFLEX_ECAPACITY
    k_ref = G.oracle_allocate(state, G.params_of(cfg, delta_cur=0))
    assert np.array_equal(k_gpu, k_ref) and ksum == int(k_ref.sum())


def test_allocate_mixed_history_and_ties():
    cfg = CFG["llada2_mini"]
    rng = np.random.default_rng(5)
    state = W.make_state(cfg, 11)
    state["hist_len"] = rng.integers(0, 3, state["hist_len"].size).astype(np.uint8)
    # quantised confidences force many equal scores
    state["conf1"] = (np.round(state["conf1"] * 8) / 8).astype(np.float32)
    state["conf2"] = (np.round(state["conf2"] * 8) / 8).astype(np.float32)
    p = G.params_of(cfg)
    k_gpu, ksum, status = G.gpu_allocate(state, p)
    assert status == B.REFLEX_OK
    assert np.array_equal(k_gpu, G.oracle_allocate(state, p))


def test_allocate_golden_worked_case():
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                    "paper_defaults.json")))["worked_allocation"]
    T = g["T"]
    state = dict(block_id=np.array(g["block_id"], np.int32),
                 seq_offsets=np.array([0, T], np.int32),
                 active_block=np.array([g["active_block"]], np.int32),
                 masked=np.array(g["masked"], np.uint8),
                 conf1=np.array(g["conf1"], np.float32),
                 conf2=np.array(g["conf1"], np.float32),
                 hist_len=np.full(T, g["hist_len"], np.uint8))
    for kmax, key in ((g["k_max_unclipped"], "expected_k_unclipped"),
                      (g["k_max_clipped"], "expected_k_clipped")):
        p = B.make_params(k_min=g["k_min"], k_max=kmax)
        k, ksum, status = G.gpu_allocate(state, p)
        assert status == B.REFLEX_OK
        assert k.tolist() == g[key]


def test_allocate_capacity_error_is_reported():
    T = 5000
    state = dict(block_id=np.ones(T, np.int32), seq_offsets=np.array([0, T], np.int32),
                 active_block=np.array([1], np.int32), masked=np.ones(T, np.uint8),
                 conf1=np.full(T, 0.5, np.float32), conf2=np.full(T, 0.5, np.float32),
                 hist_len=np.full(T, 2, np.uint8))
    k, ksum, status = G.gpu_allocate(state, B.make_params())
    assert status == B.REFLEX_ECAPACITY
    assert np.all(k == 12) and ksum == 12 * T


# ---------------------------------------------------------------------------
# the MoE layer (Eq. 2)
# ---------------------------------------------------------------------------
def _k_for(cfg, seed=0, **override):
    state = W.make_state(cfg, seed)
    return G.oracle_allocate(state, G.params_of(cfg, **override))


def test_forward_tiny_fp32_full():
    cfg = CFG["tiny_fp32"]
    layer = W.make_layer(cfg, 0)
    k = _k_for(cfg)
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(k)
    assert status == B.REFLEX_OK
    ref = G.oracle_layer(cfg, layer, k)
    G.check_routing(rec, ref, k, cfg.E)
    rel, mx = G.out_errors(out, ref["out"])
    assert rel <= G.F32_REL_L2 and mx <= G.F32_MAX_ABS, (rel, mx)


def _bf16_case(T, d, E, inter, shared, kmax, seed, weight_std=0.05):
    cfg = W.LayerConfig(name="case", dtype="bf16", d=d, E=E, inter=inter,
                        shared_inter=shared, k_min=1, k_base=min(2, kmax),
                        k_max=kmax, delta_role=1, delta_cur=1, w_cf=0.3, n_seq=1,
                        prompt_len=T, gen_len=0, block=32, weight_std=weight_std,
                        conf="uniform", mask_rule="half")
    layer = W.make_layer(cfg, seed, T=T)
    return cfg, layer


# every score-kernel band of the bf16 router (chains T x E per SM on 152 SMs)
@pytest.mark.parametrize("T,E,d", [
    (100, 64, 2048),     # ring kernel, 1 x 1 thread tiles
    (1000, 64, 2048),    # whole rows resident, ragged token tile
    (1200, 48, 512),     # whole rows resident, ragged expert tile
    (250, 256, 1024),    # whole rows resident, 4 chunks
    (700, 128, 2048),    # whole rows resident, ragged token tile, 4 expert tiles
    (2000, 32, 512),     # whole rows resident, one expert tile
    (500, 160, 1024),    # whole rows resident, 5 expert tiles, ragged expert tile
    (2000, 64, 256),     # ring kernel, 1 x 2
    (4096, 64, 256),     # ring kernel, 2 x 2, 64-k chunks
    (8192, 128, 256),    # ring kernel, 4 x 8
    (8192, 256, 256),    # ring kernel, 4 x 4
    (16384, 256, 256),   # ring kernel, 4 x 8, 4 stages
])
def test_router_scores_bit_exact_every_band(T, E, d):
    cfg, layer = _bf16_case(T, d, E, 128, 0, 8, seed=T + E + d)
    k = np.random.default_rng(T).integers(1, 9, T).astype(np.int32)
    gl = G.GpuLayer(cfg, layer)
    _, rec, status = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_ROUTE |
                                B.REFLEX_FLAG_EXACT_SCORES)
    assert status == B.REFLEX_OK
    z = oracle.router_logits(layer["hidden"], layer["w_router"])
    assert np.array_equal(rec["scores"].view(np.uint32), z.view(np.uint32))
    ids, alpha = oracle.select(z, k, cfg.k_max)
    assert np.array_equal(rec["ids"], ids)
    valid = ids >= 0
    np.testing.assert_allclose(rec["alpha"][valid], alpha[valid], rtol=G.ALPHA_RTOL, atol=1e-7)


@pytest.mark.parametrize("T,E,d", [(1000, 64, 2048), (250, 256, 1024)])
def test_router_without_renorm_bit_exact(T, E, d):
    # weights over all experts' scores (softmax over every expert)
    cfg, layer = _bf16_case(T, d, E, 128, 0, 8, seed=T + 7)
    k = np.random.default_rng(T + 2).integers(1, 9, T).astype(np.int32)
    gl = G.GpuLayer(cfg, layer)
    _, rec, status = gl.forward(k, flags=B.REFLEX_STAGE_ROUTE)
    assert status == B.REFLEX_OK
    z = oracle.router_logits(layer["hidden"], layer["w_router"])
    assert np.array_equal(rec["scores"].view(np.uint32), z.view(np.uint32))
    ids, alpha = oracle.select(z, k, cfg.k_max, renorm=False)
    assert np.array_equal(rec["ids"], ids)
    valid = ids >= 0
    np.testing.assert_allclose(rec["alpha"][valid], alpha[valid], rtol=G.ALPHA_RTOL, atol=1e-7)


def _bf16_floats(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32)


def _screen_bound(layer, d, k_splits_max=16):
    # the screen's interval half-width for every (token, expert), as the
    # kernel states it: (gamma_d + 2^-12 + (s + 1) u) ||h_t|| ||w_e||
    u = 2.0 ** -24
    g = d * u / (1 - d * u) + 2.0 ** -12 + (k_splits_max + 1) * u
    hn = np.linalg.norm(_bf16_floats(layer["hidden"]).astype(np.float64), axis=1)
    wn = np.linalg.norm(_bf16_floats(layer["w_router"]).astype(np.float64), axis=1)
    return g * np.outer(hn, wn) * 1.01


# screened routing (tensor-core scores, exact recomputation of the experts
# that could be selected): ids, alpha and the selected scores bit for bit
# (the screen runs from 128 experts and 2048 x 256 scores on; up to 256
# experts the batched recheck, above it the per-token recheck)
@pytest.mark.parametrize("T,E,d,kmax", [
    (4096, 128, 2048, 12),   # 128-wide score tiles
    (2100, 256, 1024, 12),   # ragged token tiles, two score tiles per row
    (4096, 256, 2048, 8),    # LLaDA2.0-mini expert count
    (3300, 160, 512, 6),     # ragged expert tile
    (2048, 256, 256, 4),     # short rows
    (2048, 512, 1024, 12),   # per-token recheck, split-K score slices
    (1024, 1024, 512, 8),    # per-token recheck, 1024 experts
])
def test_screened_routing_bit_exact(T, E, d, kmax):
    cfg, layer = _bf16_case(T, d, E, 128, 0, kmax, seed=3 * T + E)
    k = np.random.default_rng(T + 1).integers(1, kmax + 1, T).astype(np.int32)
    gl = G.GpuLayer(cfg, layer)
    _, rec, status = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_ROUTE)
    assert status == B.REFLEX_OK
    z = oracle.router_logits(layer["hidden"], layer["w_router"])
    ids, alpha = oracle.select(z, k, kmax)
    assert np.array_equal(rec["ids"], ids)
    valid = ids >= 0
    np.testing.assert_allclose(rec["alpha"][valid], alpha[valid], rtol=G.ALPHA_RTOL, atol=1e-7)
    rows = np.repeat(np.arange(T), kmax).reshape(T, kmax)[valid]
    got = rec["scores"][rows, ids[valid]]
    assert np.array_equal(got.view(np.uint32), z[rows, ids[valid]].view(np.uint32))
    # every other score is a tensor-core estimate inside the stated bound
    assert np.all(np.abs(rec["scores"].astype(np.float64) - z) <= _screen_bound(layer, d))


@pytest.mark.parametrize("T,E", [(4096, 128), (1000, 64), (1024, 512)])
def test_screened_routing_ties_and_many_candidates(T, E):
    # exact ties (duplicated router rows: the lower index wins), near ties
    # (rows one bf16 step apart) and 40 identical rows, more candidates than
    # one warp recomputes (every expert of such a token is recomputed); 4096
    # x 128 runs the batched recheck, 1024 x 512 the per-token recheck, 1000
    # x 64 the dense score kernels and the plain selection
    d, kmax = 1024, 8
    cfg, layer = _bf16_case(T, d, E, 128, 0, kmax, seed=99)
    w = layer["w_router"].copy()
    w[5] = w[3]
    w[9] = w[3]
    w[12] = w[11]
    w[12, 7] ^= np.uint16(1)                       # one bf16 ulp away
    w[20:60] = w[19]                               # 41 identical experts
    layer["w_router"] = w
    k = np.random.default_rng(5).integers(1, kmax + 1, T).astype(np.int32)
    gl = G.GpuLayer(cfg, layer)
    _, rec, status = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_ROUTE)
    assert status == B.REFLEX_OK
    z = oracle.router_logits(layer["hidden"], layer["w_router"])
    ids, alpha = oracle.select(z, k, kmax)
    assert np.array_equal(rec["ids"], ids)
    valid = ids >= 0
    np.testing.assert_allclose(rec["alpha"][valid], alpha[valid], rtol=G.ALPHA_RTOL, atol=1e-7)
    assert np.any(ids == 19) and not np.any(ids == 59)  # a tie group is resolved low


def test_screened_and_exact_routing_agree_on_the_whole_layer():
    cfg = CFG["llada2_mini"]
    layer = W.make_layer(cfg, 4)
    k = _k_for(cfg)
    gl = G.GpuLayer(cfg, layer)
    out_s, rec_s, st_s = gl.forward(k)
    out_e, rec_e, st_e = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK |
                                    B.REFLEX_FLAG_EXACT_SCORES)
    assert st_s == st_e == B.REFLEX_OK
    for key in ("ids", "alpha", "offsets", "perm", "row_of"):
        assert np.array_equal(rec_s[key], rec_e[key]), key
    assert np.array_equal(out_s.view(np.uint32), out_e.view(np.uint32))


# Adversarial inputs for the screen's one assumption (the tensor cores' fp32
# accumulation errs by at most 2^-12 sum_k |h_k w_k|): rows whose products
# cancel (sum |h w| far above |z|), bf16 inputs spread over many binary
# orders of magnitude, d = 4096, and the most K slices the screen takes
# (2: from 2048 x 256 scores on, the tile count leaves no room for more).
# Ids, weights and selected scores must stay bit-exact; every tensor-core
# estimate left in the record is checked against the assumed bound and the
# largest observed ratio is printed (TC_ERROR_RATIO).
def _cancelling_case(T, d, E, seed):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((T, d // 2)).astype(np.float32)
    y = (0.02 * rng.standard_normal((E, d // 2))).astype(np.float32)
    eps = (0.005 * rng.standard_normal((E, d // 2))).astype(np.float32)
    xb = W.bf16_bits_to_f32(W.to_bf16_bits(x))
    yb = W.bf16_bits_to_f32(W.to_bf16_bits(y))
    h = np.concatenate([xb, xb], axis=1)                    # [x, x]
    w = np.concatenate([yb, -yb + eps], axis=1)             # [y, -y + eps]
    return W.to_bf16_bits(h), W.to_bf16_bits(w)


def _wide_exponent_case(T, d, E, seed):
    rng = np.random.default_rng(seed)

    def spread(shape, lo, hi):
        mant = rng.uniform(1.0, 2.0, shape)
        sign = rng.choice([-1.0, 1.0], shape)
        return (sign * mant * np.exp2(rng.integers(lo, hi + 1, shape))).astype(np.float32)
    return W.to_bf16_bits(spread((T, d), -24, 8)), W.to_bf16_bits(spread((E, d), -30, 0))


@pytest.mark.parametrize("kind,T,E,d", [
    ("cancel", 4096, 128, 2048),     # 2 K slices
    ("cancel", 2048, 256, 4096),     # 2 K slices, d = 4096
    ("wide", 2048, 256, 2048),       # 2 K slices
    ("wide", 4096, 256, 4096),       # 1 slice, d = 4096
    ("gauss", 2048, 256, 4096),      # 2 K slices, d = 4096
    ("cancel", 1024, 512, 2048),     # the per-token recheck (more than 256 experts)
    ("wide", 1024, 512, 4096),       # the per-token recheck, d = 4096
])
def test_screened_routing_adversarial_inputs(kind, T, E, d):
    kmax = 8
    if kind == "cancel":
        hb, wb = _cancelling_case(T, d, E, 41)
    elif kind == "wide":
        hb, wb = _wide_exponent_case(T, d, E, 43)
    else:
        _, lay = _bf16_case(T, d, E, 128, 0, kmax, seed=45)
        hb, wb = lay["hidden"], lay["w_router"]
    cfg, layer = _bf16_case(T, d, E, 128, 0, kmax, seed=47)
    layer = dict(layer, hidden=hb, w_router=wb)
    k = np.random.default_rng(T + E).integers(1, kmax + 1, T).astype(np.int32)
    gl = G.GpuLayer(cfg, layer)
    _, rec, status = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_ROUTE)
    assert status == B.REFLEX_OK
    z = oracle.router_logits(hb, wb)
    ids, alpha = oracle.select(z, k, kmax)
    assert np.array_equal(rec["ids"], ids)
    valid = ids >= 0
    np.testing.assert_allclose(rec["alpha"][valid], alpha[valid], rtol=G.ALPHA_RTOL, atol=1e-7)
    rows = np.repeat(np.arange(T), kmax).reshape(T, kmax)[valid]
    assert np.array_equal(rec["scores"][rows, ids[valid]].view(np.uint32),
                          z[rows, ids[valid]].view(np.uint32))
    # the tensor-core estimates (entries not recomputed with the chain)
    hf = _bf16_floats(hb).astype(np.float64)
    wf = _bf16_floats(wb).astype(np.float64)
    exact = hf @ wf.T
    absdot = np.abs(hf) @ np.abs(wf).T
    est = rec["scores"].view(np.uint32) != z.view(np.uint32)
    assert est.sum() > T                     # most scores stayed estimates
    ratio = np.abs(rec["scores"].astype(np.float64) - exact)[est] / absdot[est]
    worst = float(ratio.max())
    print(f"TC_ERROR_RATIO kind={kind} T={T} E={E} d={d} max={worst:.3e} "
          f"(2^-12 = {2.0 ** -12:.3e}) median={float(np.median(ratio)):.3e} "
          f"estimates={int(est.sum())} cancellation={float(np.median(absdot / (np.abs(exact) + 1e-30))):.1f}")
    assert worst <= 2.0 ** -12


@pytest.mark.parametrize("T,E", [(4096, 256), (1024, 512)])
def test_screened_routing_router_rows_16_byte_aligned(T, E):
    # a router matrix that starts 16 bytes past a 32-byte boundary: the
    # per-token recheck (E = 512) reads expert rows with 16-byte loads
    # instead of 32-byte ones; the batched one (E = 256) stages them by TMA
    d, kmax = 2048, 8
    cfg, layer = _bf16_case(T, d, E, 128, 0, kmax, seed=51)
    gl = G.GpuLayer(cfg, layer)
    flat = torch.empty(E * d + 8, dtype=torch.bfloat16, device="cuda")
    w_off = flat[8:].view(E, d)
    w_off.copy_(gl.dev["w_router"])
    assert w_off.data_ptr() % 32 == 16
    gl.moe.w = dict(gl.moe.w, w_router=w_off)
    k = np.random.default_rng(52).integers(1, kmax + 1, T).astype(np.int32)
    _, rec, status = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_ROUTE)
    assert status == B.REFLEX_OK
    z = oracle.router_logits(layer["hidden"], layer["w_router"])
    ids, alpha = oracle.select(z, k, kmax)
    assert np.array_equal(rec["ids"], ids)
    valid = ids >= 0
    np.testing.assert_allclose(rec["alpha"][valid], alpha[valid], rtol=G.ALPHA_RTOL, atol=1e-7)


# The batched screen (bf16, renormalised weights; up to 64 experts from 8192
# tokens, 65-256 experts from 2048): tensor-core scores with the token norms
# from the same GEMM, one exact chain per candidate pair in a block of 32
# tokens (16 above 64 experts); ids, weights and selected scores bit for bit
@pytest.mark.parametrize("T,E,d,kmax", [
    (8192, 64, 2048, 12),    # whole token tiles
    (9000, 64, 1024, 8),     # ragged last tile
    (8256, 40, 512, 6),      # fewer experts than the 64-row expert box
    (8192, 64, 256, 12),     # short rows (4 chunks)
    (16384, 17, 2048, 4),    # odd expert count
    (12289, 64, 1024, 8),    # one token in the last CTA
    (30000, 48, 512, 12),    # ragged last CTA, 48 experts
    (8192, 1, 256, 1),       # a single expert: every token's one candidate
    (8200, 8, 512, 8),       # counts up to k = E
    (8192, 256, 2048, 12),   # 256 experts: eight 32-expert groups per lane
    (9000, 200, 1024, 8),    # 200 experts (a partial group), ragged last CTA
    (8192, 96, 512, 32),     # 96 experts, counts up to 32
    (16384, 256, 1024, 8),   # 256 experts, 1024 blocks
    (20000, 200, 512, 12),   # 200 experts, ragged last CTA
])
def test_batch_screened_routing_bit_exact(T, E, d, kmax):
    cfg, layer = _bf16_case(T, d, E, 128, 0, kmax, seed=5 * T + E + d)
    k = np.random.default_rng(T + E).integers(1, min(kmax, E) + 1, T).astype(np.int32)
    gl = G.GpuLayer(cfg, layer)
    _, rec, status = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_ROUTE)
    assert status == B.REFLEX_OK
    z = oracle.router_logits(layer["hidden"], layer["w_router"])
    ids, alpha = oracle.select(z, k, kmax)
    assert np.array_equal(rec["ids"], ids)
    valid = ids >= 0
    np.testing.assert_allclose(rec["alpha"][valid], alpha[valid], rtol=G.ALPHA_RTOL, atol=1e-7)
    rows = np.repeat(np.arange(T), kmax).reshape(T, kmax)[valid]
    assert np.array_equal(rec["scores"][rows, ids[valid]].view(np.uint32),
                          z[rows, ids[valid]].view(np.uint32))
    assert np.all(np.abs(rec["scores"].astype(np.float64) - z) <= _screen_bound(layer, d, 1))
    # the weights are those of the dense path, bit for bit
    _, rec_e, st_e = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_ROUTE |
                                B.REFLEX_FLAG_EXACT_SCORES)
    assert st_e == B.REFLEX_OK
    assert np.array_equal(rec["ids"], rec_e["ids"])
    assert np.array_equal(rec["alpha"].view(np.uint32), rec_e["alpha"].view(np.uint32))


@pytest.mark.parametrize("kind,E,T", [
    ("ties", 64, 8192), ("all_candidates", 64, 8192), ("cancel", 64, 8192),
    ("wide", 64, 8192),
    # above 64 experts (16-token blocks): more candidate pairs per block
    # than one pass of the chain loop, every expert row streamed again
    ("all_candidates", 256, 8192), ("ties", 256, 8192),
    ("all_candidates", 200, 16400), ("cancel", 256, 16384),
])
def test_batch_screened_routing_hard_inputs(kind, E, T):
    # ties: duplicated rows (the lower index wins), rows one bf16 step apart;
    # all_candidates: every expert row equal for 30 experts and tiny weights
    # elsewhere, so every token keeps at least 30 candidates and CTAs hold
    # more pairs than one pass of the chain loop (rows streamed again);
    # cancel / wide: the adversarial inputs of the 256-expert screen
    d, kmax = 1024, 8
    cfg, layer = _bf16_case(T, d, E, 128, 0, kmax, seed=77)
    hb, wb = layer["hidden"], layer["w_router"].copy()
    if kind == "ties":
        wb[5] = wb[3]
        wb[9] = wb[3]
        wb[12] = wb[11]
        wb[12, 7] ^= np.uint16(1)
    elif kind == "all_candidates":
        wb[:] = W.to_bf16_bits(W.bf16_bits_to_f32(wb) * np.float32(1e-3))
        wb[10:40] = wb[10]
    elif kind == "cancel":
        hb, wb = _cancelling_case(T, d, E, 78)
    else:
        hb, wb = _wide_exponent_case(T, d, E, 79)
    layer = dict(layer, hidden=hb, w_router=wb)
    k = np.random.default_rng(80).integers(1, kmax + 1, T).astype(np.int32)
    gl = G.GpuLayer(cfg, layer)
    _, rec, status = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_ROUTE)
    assert status == B.REFLEX_OK
    z = oracle.router_logits(hb, wb)
    ids, alpha = oracle.select(z, k, kmax)
    assert np.array_equal(rec["ids"], ids)
    valid = ids >= 0
    np.testing.assert_allclose(rec["alpha"][valid], alpha[valid], rtol=G.ALPHA_RTOL, atol=1e-7)
    est = rec["scores"].view(np.uint32) != z.view(np.uint32)
    if est.any():
        hf = _bf16_floats(hb).astype(np.float64)
        wf = _bf16_floats(wb).astype(np.float64)
        ratio = np.abs(rec["scores"].astype(np.float64) - hf @ wf.T)[est] / \
            (np.abs(hf) @ np.abs(wf).T)[est]
        print(f"TC_ERROR_RATIO batch kind={kind} E={E} max={float(ratio.max()):.3e} "
              f"estimates={int(est.sum())}")
        assert float(ratio.max()) <= 2.0 ** -12


@pytest.mark.parametrize("T,d,E,inter,shared,kmax,kmode", [
    (96, 256, 8, 128, 0, 4, "random"),     # one partial m-tile per expert
    (1000, 256, 4, 128, 0, 4, "max"),      # 8 m-tiles per expert, ragged tail
    (777, 512, 16, 256, 128, 6, "random"),  # shared expert, N > one tile
    (1, 256, 8, 128, 0, 4, "random"),      # single token
    (300, 256, 64, 128, 0, 2, "one"),      # many empty experts
    (500, 256, 16, 128, 0, 8, "max"),      # every token at k_max: two ragged m-tiles per group
    (1500, 256, 8, 256, 0, 4, "random"),   # CTA-pair tiles, a few hundred rows per group
    (4096, 256, 256, 512, 0, 6, "random"),  # 1-SM 256-wide tiles, ~48 rows per group
    (4096, 256, 4, 128, 0, 4, "random"),   # CTA-pair (2-SM) GEMMs, ragged groups
    (2048, 512, 8, 256, 0, 4, "max"),      # CTA-pair GEMMs, several n-tiles
    (4096, 256, 512, 64, 0, 8, "random"),  # block masks past one CTA: 32-token count + scan
    (5000, 256, 16, 128, 0, 4, "random"),  # 256-token dispatch blocks, ragged last block
    (1030, 256, 4, 128, 0, 1, "one"),      # CTA-pair tiles, ~257 rows per group: the last
                                           # tile holds a row or two (peer CTA's half empty)
    (4099, 256, 4, 128, 0, 4, "max"),      # CTA-pair tiles, T % 4 != 0, every token at k_max
    (300, 256, 1, 128, 0, 1, "one"),       # a single expert: one dense group (CTA pairs)
    (257, 256, 8, 128, 0, 8, "max"),       # every token selects every expert (k = E)
])
@pytest.mark.parametrize("simt", [False, True])
def test_forward_bf16_small(T, d, E, inter, shared, kmax, kmode, simt):
    cfg, layer = _bf16_case(T, d, E, inter, shared, kmax, seed=T + E)
    rng = np.random.default_rng(T)
    if kmode == "random":
        k = rng.integers(1, kmax + 1, T).astype(np.int32)
    elif kmode == "max":
        k = np.full(T, kmax, np.int32)
    else:
        k = np.ones(T, np.int32)
    gl = G.GpuLayer(cfg, layer)
    flags = B.REFLEX_FLAG_RENORM_TOPK | (B.REFLEX_FLAG_SIMT_EXPERTS if simt else 0)
    out, rec, status = gl.forward(k, flags=flags)
    assert status == B.REFLEX_OK
    ref = G.oracle_layer(cfg, layer, k)
    G.check_routing(rec, ref, k, cfg.E)
    rel, mx = G.out_errors(out, ref["out"])
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)


@pytest.mark.parametrize("T,d,E,inter,kmax", [
    (300, 4096, 16, 128, 8),    # d > 2048: warp-per-token combine, ring score kernel
    (512, 256, 1024, 128, 32),  # 1024 experts, k up to 32: 32 scores per lane, and
                                # screened tokens with more than 32 candidates
])
def test_forward_bf16_edges(T, d, E, inter, kmax):
    # the benchmark layers' weight scale (std 0.02), so the outputs have their
    # magnitude and the absolute bound means the same thing
    cfg, layer = _bf16_case(T, d, E, inter, 0, kmax, seed=T + d + E, weight_std=0.02)
    k = np.random.default_rng(E).integers(1, kmax + 1, T).astype(np.int32)
    k[:8] = kmax
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(k)
    assert status == B.REFLEX_OK
    ref = G.oracle_layer(cfg, layer, k)
    G.check_routing(rec, ref, k, cfg.E)
    rel, mx = G.out_errors(out, ref["out"])
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)


def test_forward_llada_moe_full():
    cfg = CFG["llada_moe"]
    layer = W.make_layer(cfg, 0)
    k = _k_for(cfg)
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(k)
    assert status == B.REFLEX_OK
    ref = G.oracle_layer(cfg, layer, k)          # every token
    G.check_routing(rec, ref, k, cfg.E)
    rel, mx = G.out_errors(out, ref["out"])
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)
    # the SIMT expert path agrees with the tensor-core path
    out2, rec2, status2 = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK |
                                     B.REFLEX_FLAG_SIMT_EXPERTS)
    assert status2 == B.REFLEX_OK
    rel2, mx2 = G.out_errors(out2, ref["out"])
    assert rel2 <= G.BF16_REL_L2 and mx2 <= G.BF16_MAX_ABS


def test_forward_llada2_mini_sampled():
    cfg = CFG["llada2_mini"]
    layer = W.make_layer(cfg, 0)
    state = W.make_state(cfg, 0)
    k = G.oracle_allocate(state, G.params_of(cfg))
    tokens = W.sample_tokens(state)
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(k)
    assert status == B.REFLEX_OK
    ref = G.oracle_layer(cfg, layer, k, tokens=tokens)
    G.check_routing(rec, ref, k, cfg.E)
    rel, mx = G.out_errors(out[tokens], ref["out"])
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)


def test_forward_fixed_counts_equal_uniform_run():
    # delta_role = delta_cur = 0 -> uniform K_base: identical to a plain
    # fixed top-K_base call on the same kernels, bit for bit
    cfg = CFG["llada_moe"]
    layer = W.make_layer(cfg, 1)
    k_alloc = _k_for(cfg, 1, delta_role=0, delta_cur=0)
    assert np.all(k_alloc == cfg.k_base)
    gl = G.GpuLayer(cfg, layer)
    a, _, _ = gl.forward(k_alloc)
    b, _, _ = gl.forward(np.full(cfg.T, cfg.k_base, np.int32))
    assert np.array_equal(a, b)


def test_forward_without_renorm():
    cfg = CFG["tiny_fp32"]
    layer = W.make_layer(cfg, 3)
    k = _k_for(cfg, 3)
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(k, flags=0)
    ref = G.oracle_layer(cfg, layer, k, renorm=False)
    G.check_routing(rec, ref, k, cfg.E)
    rel, mx = G.out_errors(out, ref["out"])
    assert rel <= G.F32_REL_L2 and mx <= G.F32_MAX_ABS


def test_smaller_batch_in_a_larger_workspace():
    # a layer sized for 513 tokens runs 512 (256 experts: the score region's
    # split count falls from 512 to 513 tokens) and matches a layer sized
    # for 512 bit for bit
    T, d, E, inter, kmax = 512, 2048, 256, 128, 8
    cfg, layer = _bf16_case(T, d, E, inter, 0, kmax, seed=41, weight_std=0.02)
    dl = api.layer_to_device(layer, cfg.dtype)
    k = torch.from_numpy(np.random.default_rng(41).integers(1, kmax + 1, T)
                         .astype(np.int32)).cuda()
    outs = []
    for max_tokens in (T, T + 1):
        moe = api.MoELayer(dl, dtype="bf16", d=d, E=E, inter=inter, shared_inter=0,
                           k_max=kmax, max_tokens=max_tokens)
        assert moe.ws_bytes >= B.reflex_moe_workspace_size(B.REFLEX_DTYPE_BF16, T, d, E,
                                                           inter, 0, kmax)
        outs.append(moe.forward(dl["hidden"], k).clone())
        torch.cuda.synchronize()
        assert moe.status() == B.REFLEX_OK
    assert torch.equal(outs[0].view(torch.int16), outs[1].view(torch.int16))


def test_forward_count_out_of_range_flagged():
    cfg = CFG["tiny_fp32"]
    layer = W.make_layer(cfg, 0)
    gl = G.GpuLayer(cfg, layer)
    k = np.full(cfg.T, 2, np.int32)
    k[5] = 9                       # > k_max
    _, rec, status = gl.forward(k)
    assert status == B.REFLEX_EKRANGE
    assert (rec["ids"][5] >= 0).sum() == cfg.k_max   # clamped, still routed


# Stages run one per call on one workspace give the bits of one call with
# every stage (1-SM tiles; CTA-pair tiles with the shared expert; the
# residual added)
@pytest.mark.parametrize("name,extra", [
    ("llada_moe", 0),
    ("llada2_mini", 0),
    ("llada_moe", B.REFLEX_FLAG_RESIDUAL),
    ("llada2_mini", B.REFLEX_FLAG_GATHER_IN_GEMM),  # DISPATCH places, EXPERT_UP gathers
])
def test_forward_stages_compose(name, extra):
    cfg = CFG[name]
    layer = W.make_layer(cfg, 2)
    k = _k_for(cfg, 2)
    gl = G.GpuLayer(cfg, layer)
    full, _, _ = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK | extra)
    kd = torch.from_numpy(k).cuda()
    out = torch.empty_like(gl.dev["hidden"])
    for st in (B.REFLEX_STAGE_ROUTE, B.REFLEX_STAGE_DISPATCH,
               B.REFLEX_STAGE_EXPERT_UP, B.REFLEX_STAGE_EXPERT_DOWN,
               B.REFLEX_STAGE_COMBINE):
        gl.moe.forward(gl.dev["hidden"], kd, out=out,
                       flags=B.REFLEX_FLAG_RENORM_TOPK | extra | st)
    torch.cuda.synchronize()
    assert np.array_equal(G.to_f32(out), full)


# ---------------------------------------------------------------------------
# fused dispatch (REFLEX_FLAG_GATHER_IN_GEMM): the CTA-pair gate/up GEMM
# fetches its rows from the token rows with four-row TMA gathers; same rows,
# tiles and MMA order as the copied rows, so the same output bits
# ---------------------------------------------------------------------------
_GATHER = B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_FLAG_GATHER_IN_GEMM


@pytest.mark.parametrize("T,d,E,inter,kmax,kmode", [
    (1500, 256, 8, 256, 4, "random"),   # a few hundred rows per group
    (4096, 256, 4, 128, 4, "random"),   # ragged groups
    (2048, 512, 8, 256, 4, "max"),      # several n-tiles
    (1030, 256, 4, 128, 1, "one"),      # last tile a row or two: clamped gathers
    (4099, 256, 4, 128, 4, "max"),      # the last token gathered, T % 4 != 0
    (300, 256, 64, 128, 2, "one"),      # 1-SM tiles: the flag changes nothing
])
def test_gather_in_gemm_gives_the_default_bits(T, d, E, inter, kmax, kmode):
    cfg, layer = _bf16_case(T, d, E, inter, 0, kmax, seed=T + E + 1)
    rng = np.random.default_rng(T + 1)
    if kmode == "random":
        k = rng.integers(1, kmax + 1, T).astype(np.int32)
    elif kmode == "max":
        k = np.full(T, kmax, np.int32)
    else:
        k = np.ones(T, np.int32)
    gl = G.GpuLayer(cfg, layer)
    out_d, _, st_d = gl.forward(k)
    out_g, rec_g, st_g = gl.forward(k, flags=_GATHER)
    assert st_d == B.REFLEX_OK and st_g == B.REFLEX_OK
    assert np.array_equal(out_g.view(np.uint32), out_d.view(np.uint32))
    ref = G.oracle_layer(cfg, layer, k)
    G.check_routing(rec_g, ref, k, cfg.E)
    rel, mx = G.out_errors(out_g, ref["out"])
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)


@pytest.mark.parametrize("name", ["llada2_mini", "llada_moe_b32"])
def test_gather_in_gemm_full_layers_give_the_default_bits(name):
    cfg = CFG[name]
    layer = W.make_layer(cfg, 3)
    k = _k_for(cfg, 3)
    gl = G.GpuLayer(cfg, layer)
    out_d, _, st_d = gl.forward(k)
    out_g, _, st_g = gl.forward(k, flags=_GATHER)
    assert st_d == B.REFLEX_OK and st_g == B.REFLEX_OK
    assert np.array_equal(out_g.view(np.uint32), out_d.view(np.uint32))


# ---------------------------------------------------------------------------
# stacked layers (shared counts, residual h <- bf16(h + MoE(h)))
# ---------------------------------------------------------------------------
def test_stack_layerwise_residual():
    """Each GPU layer runs on the oracle's input of that layer (so routing is
    comparable bit for bit in every layer); its bf16 output must match the
    oracle's residual update within the bf16 tolerance."""
    T, d, E, I, km = 256, 256, 16, 128, 4
    cfg, lay0 = _bf16_case(T, d, E, I, 0, km, seed=21)
    layers = [W.make_layer(cfg, 100 + l, T=T) for l in range(3)]
    rng = np.random.default_rng(4)
    k = rng.integers(1, km + 1, T).astype(np.int32)
    trace = oracle.moe_stack(layers[0]["hidden"], layers, k, km)
    for l, res in enumerate(trace):
        lay = dict(layers[l], hidden=res["h_in"])
        gl = G.GpuLayer(cfg, lay)
        out, rec, status = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK |
                                      B.REFLEX_FLAG_RESIDUAL)
        assert status == B.REFLEX_OK
        G.check_routing(rec, res, k, E)
        ref = W.bf16_bits_to_f32(res["h_out"]).astype(np.float64)
        rel, mx = G.out_errors(out, ref)
        assert rel <= G.BF16_REL_L2, (l, rel)
        assert G.residual_excess(out, ref, rounded_ref=True) <= 0, (l, mx)


def test_forward_llada_moe_b32_sampled():
    """One layer of the 16-layer stack at full size (32 x 1024 tokens), with
    the residual connection; routing on sampled tokens plus whole-record
    properties, outputs on sampled tokens."""
    cfg = CFG["llada_moe_b32"]
    layer = W.make_layer(cfg, 0)
    state = W.make_state(cfg, 0)
    k = G.oracle_allocate(state, G.params_of(cfg))
    tokens = W.sample_tokens(state, stride=97)
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(k, flags=B.REFLEX_FLAG_RENORM_TOPK |
                                  B.REFLEX_FLAG_RESIDUAL)
    assert status == B.REFLEX_OK
    G.check_sampled_routing(rec, layer, k, cfg.k_max, tokens)
    sub = dict(layer, hidden=layer["hidden"][tokens])
    ids, alpha = oracle.select(oracle.router_logits(sub["hidden"], layer["w_router"]),
                               k[tokens], cfg.k_max)
    ref = oracle.moe_tokens(sub["hidden"], layer["w_gate_up"], layer["w_down"], ids,
                            alpha, k[tokens], np.arange(tokens.size, dtype=np.int32))
    ref = ref + W.bf16_bits_to_f32(sub["hidden"]).astype(np.float64)
    rel, mx = G.out_errors(out[tokens], ref)
    assert rel <= G.BF16_REL_L2, rel
    assert G.residual_excess(out[tokens], ref, rounded_ref=False) <= 0, mx


def test_forward_llada_moe_b32_moe_output_sampled():
    """The same full-size layer without the residual: the MoE output itself
    (Eq. 2) on sampled tokens at the layer-output tolerance, and the whole
    routing record's properties."""
    cfg = CFG["llada_moe_b32"]
    layer = W.make_layer(cfg, 3)
    state = W.make_state(cfg, 3)
    k = G.oracle_allocate(state, G.params_of(cfg))
    tokens = W.sample_tokens(state, stride=89)
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(k)
    assert status == B.REFLEX_OK
    G.check_sampled_routing(rec, layer, k, cfg.k_max, tokens)
    h = layer["hidden"][tokens]
    ids, alpha = oracle.select(oracle.router_logits(h, layer["w_router"]), k[tokens],
                               cfg.k_max)
    ref = oracle.moe_tokens(h, layer["w_gate_up"], layer["w_down"], ids, alpha,
                            k[tokens], np.arange(tokens.size, dtype=np.int32))
    rel, mx = G.out_errors(out[tokens], ref)
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)


# ---------------------------------------------------------------------------
# token-count and count-skew sweep on the LLaDA2.0-mini layer shape
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("skew", [0.0, 0.5, 1.0])
def test_sweep_small_batch_full(skew):
    cfg = CFG["llada2_mini"]
    T = 256
    layer = W.make_layer(cfg, 7, T=T)
    k = W.skewed_k(T, skew, cfg.k_min, cfg.k_base, cfg.k_max, seed=7)
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(k)
    assert status == B.REFLEX_OK
    ref = G.oracle_layer(cfg, layer, k)
    G.check_routing(rec, ref, k, cfg.E)
    rel, mx = G.out_errors(out, ref["out"])
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)


def test_sweep_max_batch_sampled():
    cfg = CFG["llada2_mini"]
    T = 65536
    layer = W.make_layer(cfg, 8, T=T)
    k = W.skewed_k(T, 1.0, cfg.k_min, cfg.k_base, cfg.k_max, seed=8)
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(k)
    assert status == B.REFLEX_OK
    tokens = np.unique(np.concatenate([np.arange(0, T, 509), [T - 1]])).astype(np.int32)
    G.check_sampled_routing(rec, layer, k, cfg.k_max, tokens)
    ids, alpha = oracle.select(oracle.router_logits(layer["hidden"][tokens],
                                                    layer["w_router"]),
                               k[tokens], cfg.k_max)
    ref = oracle.moe_tokens(layer["hidden"][tokens], layer["w_gate_up"], layer["w_down"],
                            ids, alpha, k[tokens], np.arange(tokens.size, dtype=np.int32),
                            shared_gate_up=layer["shared_gate_up"],
                            shared_down=layer["shared_down"])
    rel, mx = G.out_errors(out[tokens], ref)
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (rel, mx)
