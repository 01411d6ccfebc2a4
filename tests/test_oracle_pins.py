"""Pins of the CPU oracle against facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than its own formula:
closed forms of Eq. 5-9, hand-worked cases (tests/golden), brute force on tiny
inputs, exact integer arithmetic, textbook error bounds and a dense
re-statement of Eq. 2 through numpy matmul.  A plausible slip in the oracle
(a dropped term, a wrong sign, a swapped index, a wrong tie rule) fails one of
them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2608_01784_gb300 import workloads as W

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                     "paper_defaults.json")))
D = GOLDEN["defaults"]
DEF = dict(theta=D["theta"], v_ref=D["v_ref"], tau=D["tau"])


def sig(x):
    return 1.0 / (1.0 + math.exp(-x))


# --------------------------------------------------------------------------
# exp (Cody-Waite + Taylor): error bound against the fp64 library exp
# --------------------------------------------------------------------------
def test_exp_within_two_ulp_of_libm():
    x = np.concatenate([np.linspace(-87.0, 88.7, 400001, dtype=np.float32),
                        np.float32([0.0, -0.0, 1.0, -1.0, 0.5, 1e-8, -1e-8])])
    y = oracle.exp_f32(x).astype(np.float64)
    ref = np.exp(x.astype(np.float64))
    ulp = np.spacing(ref.astype(np.float32)).astype(np.float64)
    assert np.all(np.abs(y - ref) <= 2.0 * ulp)


def test_exp_special_values():
    assert oracle.exp_f32([0.0])[0] == 1.0
    assert oracle.exp_f32([89.0])[0] == np.inf
    assert oracle.exp_f32([1000.0])[0] == np.inf
    assert oracle.exp_f32([-104.0])[0] == 0.0
    assert np.isnan(oracle.exp_f32([np.nan])[0])
    # subnormal range: one rounding of the exact value
    x = np.float32([-90.0, -95.0, -100.0, -103.0])
    y = oracle.exp_f32(x).astype(np.float64)
    ref = np.exp(x.astype(np.float64))
    assert np.all(np.abs(y - ref) <= 2.0 ** -149 * 2)


def test_exp_monotone():
    x = np.sort(np.random.default_rng(1).uniform(-100, 88, 200000)).astype(np.float32)
    y = oracle.exp_f32(x)
    assert np.all(np.diff(y) >= 0)


# --------------------------------------------------------------------------
# Frontier-Progress Score closed forms (Eq. 6-8)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("w", [D["w_cf_llada_moe"], D["w_cf_llada2_mini"]])
def test_fps_frontier_center(w):
    # forecast at theta - w/2 and one observation (P = 1, zero velocity):
    # F = sigma(w / (2 tau))^2
    c = D["theta"] - w / 2
    s = oracle.fps([c], [0.0], [1], w_cf=w, **DEF)[0]
    assert s == pytest.approx(sig(w / (2 * D["tau"])) ** 2, rel=2e-5)


def test_fps_frontier_edges_and_symmetry():
    w, th, tau = 0.30, D["theta"], D["tau"]
    # at chat = theta and chat = theta - w the two gates swap: sigma(w/tau)/2
    for c in (th, th - w):
        s = oracle.fps([c], [0.0], [1], w_cf=w, **DEF)[0]
        assert s == pytest.approx(0.5 * sig(w / tau), rel=2e-5)
    # F symmetric about theta - w/2
    for delta in (0.01, 0.05, 0.1, 0.2):
        a = oracle.fps([th - w / 2 + delta], [0.0], [1], w_cf=w, **DEF)[0]
        b = oracle.fps([th - w / 2 - delta], [0.0], [1], w_cf=w, **DEF)[0]
        assert a == pytest.approx(b, rel=5e-5)
    # far above the threshold the frontier gate closes
    s = oracle.fps([1.0], [1.0], [2], w_cf=w, **DEF)[0]
    assert s < sig(-(1.0 - th) / tau) * 1.0001


def test_fps_progress_half_at_vref():
    # vbar = v_ref gives P = sigma(0) = 1/2; with the forecast placed at the
    # frontier centre, S = sigma(w/2tau)^2 / 2
    w, th, vref = 0.30, D["theta"], D["v_ref"]
    c1 = th - w / 2 - vref          # chat = c1 + vbar = theta - w/2
    c2 = c1 - vref
    s = oracle.fps([c1], [c2], [2], w_cf=w, **DEF)[0]
    assert s == pytest.approx(0.5 * sig(w / (2 * D["tau"])) ** 2, rel=1e-4)


def test_fps_velocity_clip():
    # |v| beyond w/2 is clipped: P = sigma((v_ref - w/2)/tau) for a big rise
    w, tau, vref = 0.30, D["tau"], D["v_ref"]
    c1, c2 = 0.55, 0.05                           # v = 0.5 > w/2
    s = oracle.fps([c1], [c2], [2], w_cf=w, **DEF)[0]
    chat = c1 + w / 2
    F = sig((chat - D["theta"] + w) / tau) * sig((D["theta"] - chat) / tau)
    P = sig((vref - w / 2) / tau)
    assert s == pytest.approx(F * P, rel=1e-4)
    # a big drop is clipped to -w/2 and the forecast is clipped at 0
    s0 = oracle.fps([0.05], [0.9], [2], w_cf=w, **DEF)[0]
    F0 = sig((0.0 - D["theta"] + w) / tau) * sig((D["theta"] - 0.0) / tau)
    P0 = sig((vref + w / 2) / tau)
    assert s0 == pytest.approx(F0 * P0, rel=1e-3)


def test_fps_one_observation_is_frontier_only():
    # with one observation v = 0 and P = 1, regardless of c^{t-2}
    a = oracle.fps([0.7], [0.1], [1], w_cf=0.3, **DEF)[0]
    b = oracle.fps([0.7], [0.65], [1], w_cf=0.3, **DEF)[0]
    assert a == b
    F = sig((0.7 - 0.9 + 0.3) / 0.05) * sig((0.9 - 0.7) / 0.05)
    assert a == pytest.approx(F, rel=2e-5)


# --------------------------------------------------------------------------
# Allocation: hand-worked cases, role map, budget invariants, brute force
# --------------------------------------------------------------------------
def _alloc(block_id, active, masked, conf1, conf2=None, hist=2, seq_offsets=None,
           **kw):
    T = len(block_id)
    conf1 = np.asarray(conf1, np.float32)
    conf2 = conf1.copy() if conf2 is None else np.asarray(conf2, np.float32)
    hist = np.full(T, hist, np.uint8) if np.isscalar(hist) else np.asarray(hist, np.uint8)
    seq_offsets = np.array([0, T], np.int32) if seq_offsets is None else seq_offsets
    active = np.atleast_1d(np.asarray(active, np.int32))
    p = dict(k_min=2, k_base=8, k_max=14, delta_role=4, delta_cur=2, q=0.25,
             theta=0.9, w_cf=0.30, v_ref=0.01, tau=0.05)
    p.update(kw)
    return oracle.allocate(conf1, conf2, hist, np.asarray(masked, np.uint8),
                           np.asarray(block_id, np.int32), seq_offsets, active,
                           return_scores=True, **p)


def test_worked_allocation_golden():
    g = GOLDEN["worked_allocation"]
    k, _ = _alloc(g["block_id"], g["active_block"], g["masked"], g["conf1"],
                  hist=g["hist_len"], k_min=g["k_min"], k_max=g["k_max_unclipped"])
    assert k.tolist() == g["expected_k_unclipped"]
    k, _ = _alloc(g["block_id"], g["active_block"], g["masked"], g["conf1"],
                  hist=g["hist_len"], k_min=g["k_min"], k_max=g["k_max_clipped"])
    assert k.tolist() == g["expected_k_clipped"]


def test_role_map_closed_form():
    H = {int(a): b for a, b in GOLDEN["role_map"]["H"].items()}
    # 2 prompt tokens + 8 blocks of 2, nothing masked: pure role map
    block_id = [0, 0] + [b for b in range(1, 9) for _ in range(2)]
    for a in range(1, 9):
        k, _ = _alloc(block_id, a, [0] * len(block_id), [0.5] * len(block_id))
        for i, b in enumerate(block_id):
            dist = abs(b - a)
            assert k[i] == H[min(dist, 3) if dist >= 3 else dist]
    # active block 1: the prompt sits at distance 1 and gets K_base + delta_role
    k, _ = _alloc(block_id, 1, [0] * 18, [0.5] * 18)
    assert k[0] == k[1] == 12


def test_active_counts_closed_form():
    ac = GOLDEN["active_counts"]
    rng = np.random.default_rng(3)
    block_id = [0] * 4 + [1] * 32 + [2] * 32
    masked = [0] * 36 + [1] * 32
    k, _ = _alloc(block_id, 2, masked, rng.uniform(0, 1, 68))
    assert sorted(set(k[36:].tolist())) == [ac["low"], ac["mid"], ac["high"]]
    assert (k[36:] == ac["high"]).sum() == 8 and (k[36:] == ac["low"]).sum() == 8


def _random_case(rng, n_seq=3, prompt=16, blocks=6, blk=8, hist=2):
    block_id, masked, seq_off, act = [], [], [0], []
    for _ in range(n_seq):
        a = int(rng.integers(1, blocks + 1))
        act.append(a)
        block_id += [0] * prompt + [b for b in range(1, blocks + 1) for _ in range(blk)]
        masked += [0] * prompt + rng.integers(0, 2, blocks * blk).tolist()
        seq_off.append(len(block_id))
    T = len(block_id)
    c1 = rng.uniform(0, 1, T).astype(np.float32)
    c2 = np.clip(c1 - rng.uniform(-0.2, 0.2, T), 0, 1).astype(np.float32)
    h = rng.integers(0, 3, T) if hist is None else np.full(T, hist)
    return (np.array(block_id, np.int32), np.array(act, np.int32),
            np.array(masked, np.uint8), c1, c2, h.astype(np.uint8),
            np.array(seq_off, np.int32))


@pytest.mark.parametrize("seed", range(20))
def test_budget_invariants(seed):
    rng = np.random.default_rng(seed)
    bid, act, msk, c1, c2, h, so = _random_case(rng, hist=None)
    k, _ = _alloc(bid, act, msk, c1, c2, hist=h, seq_offsets=so)
    # unclipped (K_max >= K_cur + delta_cur): sum k = sum H(d)  (Eq. 5 budget
    # preserved by FGER, Eq. 9)
    Hsum = 0
    for s in range(len(act)):
        for i in range(so[s], so[s + 1]):
            dist = abs(int(bid[i]) - int(act[s]))
            Hsum += 12 if dist <= 1 else (8 if dist == 2 else 4)
        J = [i for i in range(so[s], so[s + 1]) if bid[i] == act[s] and msk[i]]
        assert sum(int(k[i]) for i in J) == len(J) * 12
    assert int(k.sum()) == Hsum
    assert k.min() >= 2 and k.max() <= 14


@pytest.mark.parametrize("seed", range(10))
def test_special_cases_fixed_and_fger_only(seed):
    rng = np.random.default_rng(100 + seed)
    bid, act, msk, c1, c2, h, so = _random_case(rng)
    # delta_role = delta_cur = 0: uniform count K_base (fixed token choice)
    k, _ = _alloc(bid, act, msk, c1, c2, seq_offsets=so, delta_role=0, delta_cur=0)
    assert np.all(k == 8)
    # FGER only (delta_role = 0): mean count exactly K_base
    k, _ = _alloc(bid, act, msk, c1, c2, seq_offsets=so, delta_role=0)
    assert int(k.sum()) == 8 * len(k)
    # RRB only (delta_cur = 0): every active token keeps K_cur
    k, _ = _alloc(bid, act, msk, c1, c2, seq_offsets=so, delta_cur=0)
    for s in range(len(act)):
        for i in range(so[s], so[s + 1]):
            if bid[i] == act[s]:
                assert k[i] == 12


def test_no_history_keeps_kcur():
    rng = np.random.default_rng(7)
    bid, act, msk, c1, c2, h, so = _random_case(rng, hist=0)
    k, s = _alloc(bid, act, msk, c1, c2, hist=0, seq_offsets=so)
    for q in range(len(act)):
        for i in range(so[q], so[q + 1]):
            if bid[i] == act[q]:
                assert k[i] == 12
    assert np.all(np.isnan(s))


@pytest.mark.parametrize("seed", range(30))
def test_grouping_brute_force(seed):
    """The (n, |J|-2n, n) grouping maximises sum_i S_i * dk_i over every
    assignment with those group sizes (distinct scores: unique maximiser)."""
    rng = np.random.default_rng(1000 + seed)
    nj = int(rng.integers(1, 9))
    block_id = [0, 0] + [1] * nj
    masked = [0, 0] + [1] * nj
    c1 = np.concatenate([[0.5, 0.5], rng.uniform(0.3, 1.0, nj)]).astype(np.float32)
    c2 = np.clip(c1 - rng.uniform(-0.2, 0.2, nj + 2), 0, 1).astype(np.float32)
    k, s = _alloc(block_id, 1, masked, c1, c2)
    S = s[2:].astype(np.float64)
    if len(set(S.tolist())) < nj:
        pytest.skip("tied scores drawn")
    n = math.floor(0.25 * nj)
    best, best_val = None, -np.inf
    for plus in itertools.combinations(range(nj), n):
        rest = [i for i in range(nj) if i not in plus]
        for minus in itertools.combinations(rest, n):
            dk = np.zeros(nj)
            dk[list(plus)] = 2
            dk[list(minus)] = -2
            v = float((S * dk).sum())
            if v > best_val:
                best, best_val = dk, v
    assert (k[2:] - 12).tolist() == best.astype(int).tolist()


def test_grouping_ties_lower_position_first():
    # identical confidences -> identical scores: positions decide
    block_id = [0] + [1] * 8
    masked = [0] + [1] * 8
    k, s = _alloc(block_id, 1, masked, [0.7] * 9)
    assert len(set(s[1:].tolist())) == 1
    assert k[1:].tolist() == [14, 14, 12, 12, 12, 12, 10, 10]


def test_group_size_floor():
    for nj, n in [(1, 0), (3, 0), (4, 1), (7, 1), (8, 2), (11, 2), (12, 3)]:
        k, _ = _alloc([0] + [1] * nj, 1, [0] + [1] * nj,
                      np.linspace(0.3, 0.95, nj + 1))
        assert int((k[1:] == 14).sum()) == n and int((k[1:] == 10).sum()) == n


def test_clip_bounds():
    rng = np.random.default_rng(11)
    bid, act, msk, c1, c2, h, so = _random_case(rng)
    k, _ = _alloc(bid, act, msk, c1, c2, seq_offsets=so, k_min=5, k_max=12)
    assert k.min() >= 5 and k.max() <= 12
    k2, _ = _alloc(bid, act, msk, c1, c2, seq_offsets=so, k_min=2, k_max=14)
    assert np.array_equal(np.clip(k2, 5, 12), k)


def test_role_shuffle_preserves_pairs():
    # Role-Shuffled RRB (Appendix C) keeps the count multiset: pairs = sum k
    rng = np.random.default_rng(5)
    cfg = W.CONFIGS["tiny_fp32"]
    lay = W.make_layer(cfg, 0)
    k = rng.integers(1, 5, cfg.T).astype(np.int32)
    ks = rng.permutation(k)
    for kk in (k, ks):
        z = oracle.router_logits(lay["hidden"], lay["w_router"])
        ids, _ = oracle.select(z, kk, 4)
        off, perm, row_of = oracle.permutation(ids, kk, cfg.E)
        assert perm.size == off[-1] == int(kk.sum()) == int(k.sum())


# --------------------------------------------------------------------------
# App. C ablations: rank keys of the Eq. 9 groups and Role-Shuffled RRB
# --------------------------------------------------------------------------
def _grid(x):
    """Values on a 2^-8 grid, so c1 - c2 and c1 + vbar are exact in fp32."""
    return np.round(np.asarray(x, np.float64) * 256) / 256


def _expected_groups(order, nj, q=0.25, k_cur=12, dc=2):
    """Counts of J_h members listed in rank order (first = highest key)."""
    n = math.floor(q * nj)
    k = np.full(nj, k_cur)
    k[order[:n]] += dc
    if n:
        k[order[nj - n:]] -= dc
    return k


def _active_case(c1, c2, hist):
    nj = len(c1)
    bid = [0, 0] + [1] * nj
    msk = [0, 0] + [1] * nj
    c1 = np.concatenate([[0.5, 0.5], c1]).astype(np.float32)
    c2 = np.concatenate([[0.5, 0.5], c2]).astype(np.float32)
    hist = np.concatenate([[2, 2], hist]).astype(np.uint8)
    return bid, msk, c1, c2, hist


def test_signal_frontier_orders_by_distance_to_gate_midpoint():
    # F(c) = sig((c - theta + w) / tau) * sig((theta - c) / tau) is symmetric
    # about c = theta - w/2 and falls with the distance from it (the two
    # arguments sum to w / tau), so "F only" ranks J_h by |chat - (theta - w/2)|.
    w = 0.30
    chat = _grid([0.75, 0.70, 0.82, 0.60, 0.95, 0.40, 0.78, 0.30])
    v = _grid([0.10, -0.12, 0.0, 0.05, -0.05, 0.14, -0.02, 0.08])  # |v| < w/2
    c1 = chat - v
    c2 = c1 - v
    bid, msk, C1, C2, H = _active_case(c1, c2, np.full(8, 2))
    k, key = _alloc(bid, 1, msk, C1, C2, hist=H, signal=1, w_cf=w)
    order = np.argsort(np.abs(chat - (0.9 - w / 2)), kind="stable")
    assert k[2:].tolist() == _expected_groups(order, 8).tolist()
    # the same tokens under FPS rank differently (the progress factor matters)
    k_fps, _ = _alloc(bid, 1, msk, C1, C2, hist=H, signal=0, w_cf=w)
    assert k_fps[2:].tolist() != k[2:].tolist()


def test_signal_progress_orders_single_observation_then_slowest():
    # P = sig((v_ref - vbar) / tau) falls with vbar; one observation gives 1,
    # above any value of sig at the clipped velocities (vbar >= -w/2).
    v = _grid([0.10, -0.12, 0.0, 0.05, -0.05, 0.14, -0.02, 0.08])
    hist = np.array([2, 2, 1, 2, 2, 2, 1, 2])
    c1 = _grid([0.6, 0.3, 0.9, 0.5, 0.7, 0.4, 0.2, 0.8])
    c2 = c1 - v
    bid, msk, C1, C2, H = _active_case(c1, c2, hist)
    k, _ = _alloc(bid, 1, msk, C1, C2, hist=H, signal=2)
    keyv = np.where(hist >= 2, v, -1.0)   # single observation first
    order = np.lexsort((np.arange(8), keyv))
    assert k[2:].tolist() == _expected_groups(order, 8).tolist()


@pytest.mark.parametrize("signal,sign", [(3, -1), (4, 1)])
def test_signal_confidence_and_uncertainty_are_plain_sorts(signal, sign):
    c1 = _grid([0.6, 0.3, 0.9, 0.5, 0.7, 0.4, 0.2, 0.8, 0.55, 0.35, 0.65, 0.45])
    c2 = _grid(np.clip(c1 - 0.1, 0, 1))
    bid, msk, C1, C2, H = _active_case(c1, c2, np.full(12, 2))
    k, _ = _alloc(bid, 1, msk, C1, C2, hist=H, signal=signal)
    order = np.argsort(sign * c1, kind="stable")   # confidence: high first
    assert k[2:].tolist() == _expected_groups(order, 12).tolist()


def test_signal_ties_keep_lower_position_first():
    c1 = _grid([0.7] * 8)
    bid, msk, C1, C2, H = _active_case(c1, c1, np.full(8, 2))
    for signal in range(5):
        k, _ = _alloc(bid, 1, msk, C1, C2, hist=H, signal=signal)
        assert k[2:].tolist() == [14, 14, 12, 12, 12, 12, 10, 10]


@pytest.mark.parametrize("seed", range(5))
def test_role_shuffle_keeps_each_sequence_multiset(seed):
    rng = np.random.default_rng(300 + seed)
    bid, act, msk, c1, c2, h, so = _random_case(rng, hist=None)
    for kw in (dict(delta_cur=0), dict()):   # Role-Shuffled RRB, and REFLEX
        k0, _ = _alloc(bid, act, msk, c1, c2, hist=h, seq_offsets=so, **kw)
        k1, _ = _alloc(bid, act, msk, c1, c2, hist=h, seq_offsets=so,
                       role_shuffle=1, shuffle_seed=seed, **kw)
        for s in range(len(act)):
            a, b = so[s], so[s + 1]
            assert sorted(k0[a:b].tolist()) == sorted(k1[a:b].tolist())
        assert not np.array_equal(k0, k1)
        k2, _ = _alloc(bid, act, msk, c1, c2, hist=h, seq_offsets=so,
                       role_shuffle=1, shuffle_seed=seed, **kw)
        assert np.array_equal(k1, k2)              # deterministic per seed


def test_role_shuffle_uniform_fixed_counts_untouched():
    # a uniform allocation is a fixed point of any permutation
    rng = np.random.default_rng(9)
    bid, act, msk, c1, c2, h, so = _random_case(rng)
    k, _ = _alloc(bid, act, msk, c1, c2, seq_offsets=so, delta_role=0,
                  delta_cur=0, role_shuffle=1, shuffle_seed=77)
    assert np.all(k == 8)


def test_role_shuffle_is_uniform_over_seeds():
    # 6 positions (prompt, blocks 1..5 with block 3 active: role counts 4, 8,
    # 12, 12, 12, 8 by Eq. 5): every position receives count v with frequency
    # (multiplicity of v) / 6 over seeds; chi-square with 6 x (values - 1)
    # degrees of freedom.
    bid = [0, 1, 2, 3, 4, 5]
    act, msk = 3, [0] * 6
    c1 = np.full(6, 0.5, np.float32)
    base, _ = _alloc(bid, act, msk, c1, delta_cur=0)
    vals, mult = np.unique(base, return_counts=True)
    n_seeds = 3000
    hits = np.zeros((6, len(vals)))
    for seed in range(n_seeds):
        k, _ = _alloc(bid, act, msk, c1, delta_cur=0, role_shuffle=1, shuffle_seed=seed)
        for pos in range(6):
            hits[pos, np.searchsorted(vals, k[pos])] += 1
    expect = n_seeds * mult[None, :] / 6.0
    chi2 = float(((hits - expect) ** 2 / expect).sum())
    dof = 6 * (len(vals) - 1)
    assert chi2 < dof + 6 * math.sqrt(2 * dof)     # far inside the upper tail


def test_role_shuffle_follows_key_order():
    # definition check of the assignment: token i takes the count of place
    # rank(key_i, i) in the sequence (keys from the generator, numpy sort)
    rng = np.random.default_rng(21)
    bid, act, msk, c1, c2, h, so = _random_case(rng, n_seq=2)
    k0, _ = _alloc(bid, act, msk, c1, c2, seq_offsets=so, delta_cur=0)
    seed = 123456789
    k1, _ = _alloc(bid, act, msk, c1, c2, seq_offsets=so, delta_cur=0,
                   role_shuffle=1, shuffle_seed=seed)
    for s in range(len(act)):
        a, b = int(so[s]), int(so[s + 1])
        keys = np.array([oracle.splitmix64(seed, i + 1) >> 32 for i in range(a, b)],
                        np.uint64)
        ranks = np.empty(b - a, np.int64)
        ranks[np.lexsort((np.arange(b - a), keys))] = np.arange(b - a)
        assert k1[a:b].tolist() == k0[a:b][ranks].tolist()


def test_splitmix64_matches_published_reference_outputs():
    # SplitMix64 (Steele, Lea and Flood 2014) as published: the outputs of its
    # public-domain reference implementation for two seeds
    # (tests/golden/splitmix64_reference.json).  A wrong gamma, multiplier or
    # shift in the oracle's generator fails here.
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                    "splitmix64_reference.json")))
    for v in g["vectors"]:
        seed = int(v["seed"])
        want = ([int(x, 16) for x in v["outputs_hex"]] if "outputs_hex" in v
                else [int(x) for x in v["outputs_dec"]])
        got = [oracle.splitmix64(seed, n) for n in range(1, len(want) + 1)]
        assert got == want, (seed, [hex(x) for x in got])


def test_splitmix64_bits_are_uniform_and_mix():
    out = np.array([oracle.splitmix64(42, n) for n in range(1, 1 << 15)], np.uint64)
    top = (out >> np.uint64(56)).astype(np.int64)
    hist = np.bincount(top, minlength=256)
    e = out.size / 256
    chi2 = float(((hist - e) ** 2 / e).sum())
    assert chi2 < 255 + 6 * math.sqrt(2 * 255)
    # neighbouring counters differ in about half of the 64 bits
    diff = [bin(int(a) ^ int(b)).count("1") for a, b in zip(out[:-1], out[1:])]
    assert 30 < float(np.mean(diff)) < 34
    assert len(set(out.tolist())) == out.size


# --------------------------------------------------------------------------
# Router scores: exact integer cases, summation order, fma, error bound
# --------------------------------------------------------------------------
def test_router_logits_exact_integers():
    rng = np.random.default_rng(0)
    h = rng.integers(-8, 9, (5, 64)).astype(np.float32)
    w = rng.integers(-8, 9, (7, 64)).astype(np.float32)
    z = oracle.router_logits(h, w)
    assert np.array_equal(z, (h.astype(np.int64) @ w.astype(np.int64).T).astype(np.float32))
    # bf16 inputs widen exactly
    hb, wb = W.to_bf16_bits(h), W.to_bf16_bits(w)
    assert np.array_equal(oracle.router_logits(hb, wb), z)


def test_router_logits_sequential_order():
    d = 64
    eps = np.float32(2.0 ** -24)
    h = np.full((2, d), eps, np.float32)
    h[0, 0] = 1.0          # big term first: every later half-ulp add rounds away
    h[1, -1] = 1.0         # big term last: the small ones accumulate first
    w = np.ones((1, d), np.float32)
    z = oracle.router_logits(h, w)
    assert z[0, 0] == np.float32(1.0)
    assert z[1, 0] == np.float32(1.0 + (d - 1) * 2.0 ** -24)


def test_router_logits_uses_fused_multiply_add():
    a = np.float32(1.0 + 2.0 ** -12)
    h = np.array([[a, a]], np.float32)
    w = np.array([[a, -a]], np.float32)
    z = oracle.router_logits(h, w)
    # fma keeps the exact product a*a = 1 + 2^-11 + 2^-24 in the second step
    assert z[0, 0] == np.float32(-(2.0 ** -24))


def test_router_logits_error_bound():
    rng = np.random.default_rng(2)
    h = rng.standard_normal((16, 2048)).astype(np.float32)
    w = (0.02 * rng.standard_normal((32, 2048))).astype(np.float32)
    z = oracle.router_logits(h, w).astype(np.float64)
    exact = h.astype(np.float64) @ w.astype(np.float64).T
    n, u = 2048, 2.0 ** -24
    gamma = n * u / (1 - n * u)
    bound = gamma * (np.abs(h.astype(np.float64)) @ np.abs(w.astype(np.float64)).T)
    assert np.all(np.abs(z - exact) <= bound)


# --------------------------------------------------------------------------
# TopK and router weights
# --------------------------------------------------------------------------
@pytest.mark.parametrize("seed", range(10))
def test_topk_brute_force(seed):
    rng = np.random.default_rng(seed)
    T, E, kmax = 40, 8, 4
    z = rng.integers(-3, 4, (T, E)).astype(np.float32)   # many ties
    k = rng.integers(1, kmax + 1, T).astype(np.int32)
    ids, alpha = oracle.select(z, k, kmax)
    for t in range(T):
        winners = []
        for sub in itertools.combinations(range(E), int(k[t])):
            rest = [e for e in range(E) if e not in sub]
            ok = all((z[t, a] > z[t, b]) or (z[t, a] == z[t, b] and a < b)
                     for a in sub for b in rest)
            if ok:
                winners.append(set(sub))
        assert len(winners) == 1
        assert set(ids[t, :k[t]].tolist()) == winners[0]
        # slots are in rank order
        for j in range(k[t] - 1):
            a, b = ids[t, j], ids[t, j + 1]
            assert z[t, a] > z[t, b] or (z[t, a] == z[t, b] and a < b)
        assert np.all(ids[t, k[t]:] == -1) and np.all(alpha[t, k[t]:] == 0)


def test_alpha_closed_forms():
    z = np.zeros((1, 8), np.float32)
    k = np.array([3], np.int32)
    ids, a = oracle.select(z, k, 4, renorm=True)
    assert ids[0, :3].tolist() == [0, 1, 2]
    assert np.allclose(a[0, :3], 1 / 3, rtol=0, atol=1e-15)
    ids, a = oracle.select(z, k, 4, renorm=False)
    assert np.allclose(a[0, :3], 1 / 8, rtol=0, atol=1e-15)
    z = np.array([[2.0, 0.0, 1.0, -1.0]], np.float32)
    ids, a = oracle.select(z, np.array([2], np.int32), 2, renorm=True)
    assert ids[0].tolist() == [0, 2]
    assert a[0, 0] / a[0, 1] == pytest.approx(math.e, rel=1e-12)
    assert a[0].sum() == pytest.approx(1.0, rel=1e-15)


def test_select_rejects_bad_k():
    z = np.zeros((2, 8), np.float32)
    with pytest.raises(ValueError):
        oracle.select(z, np.array([1, 5], np.int32), 4)
    with pytest.raises(ValueError):
        oracle.select(z, np.array([0, 1], np.int32), 4)


# --------------------------------------------------------------------------
# Pair permutation
# --------------------------------------------------------------------------
@pytest.mark.parametrize("seed", range(5))
def test_permutation_properties(seed):
    rng = np.random.default_rng(seed)
    T, E, kmax = 200, 16, 6
    k = rng.integers(1, kmax + 1, T).astype(np.int32)
    ids = np.full((T, kmax), -1, np.int32)
    for t in range(T):
        ids[t, :k[t]] = rng.permutation(E)[:k[t]]
    off, perm, row_of = oracle.permutation(ids, k, E)
    assert perm.size == off[E] == k.sum()              # pairs = sum k
    for e in range(E):
        rows = perm[off[e]:off[e + 1]]
        assert np.all(ids.ravel()[rows] == e)
        assert np.all(np.diff(rows // kmax) > 0)       # token order within expert
        assert off[e + 1] - off[e] == int((ids == e).sum())
    for t in range(T):
        for j in range(kmax):
            if j < k[t]:
                assert perm[row_of[t, j]] == t * kmax + j
            else:
                assert row_of[t, j] == -1


# --------------------------------------------------------------------------
# Eq. 2 layer: reductions to a plain FFN and a dense masked restatement
# --------------------------------------------------------------------------
def _ffn(h, wgu, wd):
    I = wd.shape[-1]
    g = h @ wgu[:I].T
    u = h @ wgu[I:].T
    return ((g / (1 + np.exp(-g))) * u) @ wd.T


def _small_layer(rng, T=24, d=32, E=6, I=16, s=0):
    h = rng.standard_normal((T, d)).astype(np.float32)
    wr = (0.3 * rng.standard_normal((E, d))).astype(np.float32)
    wgu = (0.2 * rng.standard_normal((E, 2 * I, d))).astype(np.float32)
    wd = (0.2 * rng.standard_normal((E, d, I))).astype(np.float32)
    sh = None
    if s:
        sh = ((0.2 * rng.standard_normal((2 * s, d))).astype(np.float32),
              (0.2 * rng.standard_normal((d, s))).astype(np.float32))
    return h, wr, wgu, wd, sh


def test_layer_single_expert_is_ffn():
    rng = np.random.default_rng(0)
    h, wr, wgu, wd, _ = _small_layer(rng, E=1)
    k = np.ones(h.shape[0], np.int32)
    res = oracle.moe_layer(h, wr, wgu, wd, k, 1)
    assert np.allclose(res["out"], _ffn(h.astype(np.float64), wgu[0].astype(np.float64),
                                        wd[0].astype(np.float64)), rtol=1e-12, atol=1e-12)


def test_layer_identical_experts_ignore_routing():
    rng = np.random.default_rng(1)
    h, wr, wgu, wd, _ = _small_layer(rng)
    wgu[:] = wgu[0]
    wd[:] = wd[0]
    k = rng.integers(1, 5, h.shape[0]).astype(np.int32)
    res = oracle.moe_layer(h, wr, wgu, wd, k, 4)
    ref = _ffn(h.astype(np.float64), wgu[0].astype(np.float64), wd[0].astype(np.float64))
    assert np.allclose(res["out"], ref, rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("renorm", [True, False])
def test_layer_matches_dense_masked_form(renorm):
    rng = np.random.default_rng(2)
    h, wr, wgu, wd, sh = _small_layer(rng, s=8)
    k = rng.integers(1, 5, h.shape[0]).astype(np.int32)
    res = oracle.moe_layer(h, wr, wgu, wd, k, 4, renorm=renorm,
                           shared_gate_up=sh[0], shared_down=sh[1])
    hd = h.astype(np.float64)
    # dense: every expert on every token, weighted by a masked weight matrix
    E = wr.shape[0]
    z = res["z"].astype(np.float64)                 # pinned separately above
    p = np.exp(z - z.max(1, keepdims=True))
    p /= p.sum(1, keepdims=True)
    mask = np.zeros_like(p)
    for t in range(h.shape[0]):
        order = sorted(range(E), key=lambda e: (-z[t, e], e))[:k[t]]
        mask[t, order] = 1
    gate = p * mask
    if renorm:
        gate /= gate.sum(1, keepdims=True)
    dense = sum(gate[:, e:e + 1] * _ffn(hd, wgu[e].astype(np.float64),
                                         wd[e].astype(np.float64)) for e in range(E))
    dense += _ffn(hd, sh[0].astype(np.float64), sh[1].astype(np.float64))
    assert np.allclose(res["out"], dense, rtol=1e-10, atol=1e-11)


def test_layer_token_subset_is_exact():
    rng = np.random.default_rng(3)
    h, wr, wgu, wd, _ = _small_layer(rng)
    k = rng.integers(1, 5, h.shape[0]).astype(np.int32)
    full = oracle.moe_layer(h, wr, wgu, wd, k, 4)
    sub = np.array([3, 0, 17], np.int32)
    part = oracle.moe_layer(h, wr, wgu, wd, k, 4, tokens=sub)
    assert np.array_equal(part["out"], full["out"][sub])


def test_layer_bf16_inputs_widen_exactly():
    rng = np.random.default_rng(4)
    h, wr, wgu, wd, _ = _small_layer(rng)
    hb, wrb, gub, db = (W.to_bf16_bits(x) for x in (h, wr, wgu, wd))
    k = rng.integers(1, 5, h.shape[0]).astype(np.int32)
    a = oracle.moe_layer(hb, wrb, gub, db, k, 4)
    b = oracle.moe_layer(W.bf16_bits_to_f32(hb), W.bf16_bits_to_f32(wrb),
                         W.bf16_bits_to_f32(gub), W.bf16_bits_to_f32(db), k, 4)
    for key in ("z", "ids", "alpha", "perm", "out"):
        assert np.array_equal(a[key], b[key])


# --------------------------------------------------------------------------
# bf16 rounding and the stacked-layer residual (reading: h <- bf16(h + out))
# --------------------------------------------------------------------------
def test_bf16_rounding_ties_and_library_agreement():
    # halfway cases round to the even significand
    one = 1.0
    cases = [(one, 0x3F80), (one + 2.0 ** -8, 0x3F80), (one + 3 * 2.0 ** -8, 0x3F82),
             (one + 2.0 ** -7, 0x3F81), (-(one + 2.0 ** -8), 0xBF80), (0.0, 0x0000),
             (-0.0, 0x8000), (3.0, 0x4040)]
    got = oracle.bf16_from_f64(np.array([c[0] for c in cases]))
    assert got.tolist() == [c[1] for c in cases]
    # fp32-representable values: agrees with torch's float -> bfloat16
    x = np.random.default_rng(0).standard_normal(100000).astype(np.float32)
    x = np.concatenate([x, x * 1e-20, x * 1e20])
    assert np.array_equal(oracle.bf16_from_f64(x.astype(np.float64)), W.to_bf16_bits(x))


def test_residual_update_closed_form():
    h = W.to_bf16_bits(np.array([1.0, -2.0, 0.5, 3.0], np.float32))
    out = np.array([0.25, 2.0, -0.5, 2.0 ** -9], np.float64)
    nxt = W.bf16_bits_to_f32(oracle.residual_bf16(h, out))
    assert nxt.tolist() == [1.25, 0.0, 0.0, 3.0]


def test_stack_shares_counts_and_chains_inputs():
    rng = np.random.default_rng(9)
    T, d, E, I = 16, 32, 4, 16
    h0 = W.to_bf16_bits(rng.standard_normal((T, d)).astype(np.float32))
    layers = []
    for _ in range(3):
        layers.append(dict(
            w_router=W.to_bf16_bits((0.3 * rng.standard_normal((E, d))).astype(np.float32)),
            w_gate_up=W.to_bf16_bits((0.2 * rng.standard_normal((E, 2 * I, d))).astype(np.float32)),
            w_down=W.to_bf16_bits((0.2 * rng.standard_normal((E, d, I))).astype(np.float32))))
    k = rng.integers(1, 3, T).astype(np.int32)
    tr = oracle.moe_stack(h0, layers, k, 2)
    assert np.array_equal(tr[0]["h_in"], h0)
    for a, b in zip(tr[:-1], tr[1:]):
        assert np.array_equal(a["h_out"], b["h_in"])
    for res in tr:
        assert res["perm"].size == int(k.sum())          # same counts per layer
    # a layer with zero down-projection leaves the stream unchanged
    zero = dict(layers[0], w_down=np.zeros_like(layers[0]["w_down"]))
    tr0 = oracle.moe_stack(h0, [zero], k, 2)
    assert np.array_equal(tr0[0]["h_out"], h0)


# --------------------------------------------------------------------------
# Score-based count rules of the threshold-based comparison methods (App. B):
# Top-p = the smallest router-ranked prefix whose routing mass reaches p;
# Expert-Threshold = the experts whose routing mass exceeds a threshold.
# --------------------------------------------------------------------------
def _softmax64(z):
    z = np.asarray(z, np.float64)
    e = np.exp(z - z.max(axis=1, keepdims=True))
    return e / e.sum(axis=1, keepdims=True)


@pytest.mark.parametrize("E", [8, 64])
def test_rule_counts_uniform_scores_closed_form(E):
    # equal scores: every expert has mass 1/E exactly (u_e = exp(0) = 1,
    # S = E), so Top-p takes ceil(p E) experts and the threshold rule takes
    # all of them below 1/E and none at or above it (then the clip)
    z = np.full((1, E), 0.375, np.float32)
    for j in (1, 3, E // 2, E):
        p = j / E
        assert oracle.rule_counts(z, 1, p, 1, E)[0] == j
        assert oracle.rule_counts(z, 1, p - 0.5 / E, 1, E)[0] == j
    assert oracle.rule_counts(z, 2, 0.99 / E, 1, 12)[0] == min(E, 12)
    assert oracle.rule_counts(z, 2, 1.0 / E, 1, 12)[0] == 1
    assert oracle.rule_counts(z, 2, 1.0 / E, 3, 12)[0] == 3


def test_rule_counts_brute_force_over_subsets():
    # E = 8: Top-p's count is the size of the smallest expert SUBSET whose
    # mass reaches p (the top-j prefix is the heaviest j-subset), found by
    # enumerating all 255 subsets in fp64; the threshold count is the number
    # of experts above the threshold in fp64.  Tokens whose fp64 masses lie
    # within 1e-5 of the threshold are left out (the oracle decides in fp32).
    rng = np.random.default_rng(17)
    T, E = 3000, 8
    z = (rng.standard_normal((T, E)) * rng.uniform(0.2, 3.0, (T, 1))).astype(np.float32)
    P = _softmax64(z)
    masks = np.array([[(s >> e) & 1 for e in range(E)] for s in range(1, 1 << E)],
                     np.float64)
    sizes = masks.sum(axis=1)
    mass = P @ masks.T                       # [T, 255] mass of every subset
    checked = 0
    for p in (0.15, 0.2, 0.5, 0.8, 0.95):
        k = oracle.rule_counts(z, 1, p, 1, E)
        ok = np.all(np.abs(mass - p) > 1e-5, axis=1)
        want = np.where(mass >= p, sizes[None, :], E + 1).min(axis=1)
        assert np.array_equal(k[ok], want[ok].astype(np.int32)), p
        checked += int(ok.sum())
    for thr in (0.05, 0.1, 0.125, 0.2, 0.4):
        k = oracle.rule_counts(z, 2, thr, 1, E)
        ok = np.all(np.abs(P - thr) > 1e-6, axis=1)
        want = np.clip((P > thr).sum(axis=1), 1, E)
        assert np.array_equal(k[ok], want[ok].astype(np.int32)), thr
        checked += int(ok.sum())
    assert checked > 0.99 * 10 * T


def test_rule_counts_one_dominant_expert_and_monotone():
    rng = np.random.default_rng(3)
    z = np.zeros((1, 64), np.float32)
    z[0, 17] = 12.0                          # mass 0.99..: one expert suffices
    assert oracle.rule_counts(z, 1, 0.9, 1, 12)[0] == 1
    assert oracle.rule_counts(z, 2, 0.01, 1, 12)[0] == 1
    assert oracle.rule_counts(z, 1, 0.9, 2, 12)[0] == 2          # k_min clip
    z = rng.standard_normal((500, 64)).astype(np.float32)
    ps = [0.05, 0.15, 0.2, 0.3, 0.6, 0.9]
    kp = np.stack([oracle.rule_counts(z, 1, p, 1, 12) for p in ps])
    assert np.all(np.diff(kp, axis=0) >= 0)          # more mass, more experts
    ts = [0.005, 0.0156, 0.019, 0.0215, 0.03, 0.08]
    kt = np.stack([oracle.rule_counts(z, 2, t, 1, 12) for t in ts])
    assert np.all(np.diff(kt, axis=0) <= 0)          # higher bar, fewer experts
    assert kp.min() >= 1 and kp.max() <= 12 and kt.min() >= 1 and kt.max() <= 12
    # p above the total mass: the upper clip
    assert np.all(oracle.rule_counts(z, 1, 1.5, 1, 12) == 12)


def test_rule_counts_route_the_selected_prefix():
    # the count and the selection agree: the top-k ids of the oracle's
    # selection with the Top-p counts carry at least mass p (fp64), and one
    # fewer expert carries less (away from the boundary)
    rng = np.random.default_rng(8)
    z = (rng.standard_normal((400, 64)) * 1.5).astype(np.float32)
    P = _softmax64(z)
    k = oracle.rule_counts(z, 1, 0.3, 1, 64)
    ids, _ = oracle.select(z, k, 64)
    for t in range(z.shape[0]):
        sel = ids[t, :k[t]]
        m = P[t, sel].sum()
        if abs(m - 0.3) > 1e-5 and abs(m - P[t, sel[-1]] - 0.3) > 1e-5:
            assert m >= 0.3 and (k[t] == 1 or m - P[t, sel[-1]] < 0.3)
