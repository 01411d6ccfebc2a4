"""Pins of the oracle's refinement-state update (Sec. 3.1, Eq. 1) and of the
trajectory driver, on CPU: a hand-worked trajectory (tests/golden), the
commit rule's set-level invariants, the history shift, block advance and
finish, termination bounds, and the closed form of the pair count under
fixed counts."""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2608_01784_gb300 import trajectory as TR
from paper_2608_01784_gb300 import workloads as W
from tests import trajectory_cases as TC

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                   "trajectory_worked.json")))


def _golden_state():
    bid = np.array(GOLD["block_id"], np.int32)
    T = bid.size
    return dict(conf1=np.zeros(T, np.float32), conf2=np.zeros(T, np.float32),
                hist_len=np.zeros(T, np.uint8), masked=(bid > 0).astype(np.uint8),
                block_id=bid, seq_offsets=np.array([0, T], np.int32),
                active_block=np.array([1], np.int32))


def test_golden_worked_trajectory():
    st = _golden_state()
    nb = np.array([GOLD["num_blocks"]], np.int32)
    for f in GOLD["forwards"]:
        st, committed = oracle.update_state(st, np.array(f["conf"], np.float32), nb,
                                            GOLD["theta"])
        assert st["masked"].tolist() == f["masked_after"], f["why"]
        assert int(st["active_block"][0]) == f["active_after"], f["why"]
        assert int(committed[0]) == f["committed"], f["why"]
        if "conf1_after" in f:
            assert np.array_equal(st["conf1"], np.array(f["conf1_after"], np.float32))
            assert np.array_equal(st["conf2"], np.array(f["conf2_after"], np.float32))
            assert st["hist_len"].tolist() == f["hist_after"]


def _random_state(seed, cfg="llada2_mini"):
    c = W.CONFIGS[cfg]
    st = W.make_state(c, seed, hist_len=None)
    rng = np.random.default_rng(seed)
    st["hist_len"] = rng.integers(0, 3, st["hist_len"].size).astype(np.uint8)
    conf = rng.uniform(0.5, 1.0, st["block_id"].size).astype(np.float32)
    return st, conf


@pytest.mark.parametrize("seed", range(8))
def test_commit_rule_set_invariants(seed):
    st, conf = _random_state(seed)
    nb = TR.num_blocks(st)
    theta = 0.9
    new, committed = oracle.update_state(st, conf, nb, theta)
    so = st["seq_offsets"]
    for s in range(nb.size):
        a = int(st["active_block"][s])
        seg = slice(so[s], so[s + 1])
        bid, m0, m1 = st["block_id"][seg], st["masked"][seg], new["masked"][seg]
        J = (m0 == 1) & (bid == a)
        C = (m0 == 1) & (m1 == 0)
        assert not np.any(C & ~J)                       # commits only in J
        assert np.all(m1[~J] == m0[~J])                 # everything else kept
        above = J & (conf[seg] >= theta)
        if above.any():
            assert np.array_equal(C, above)             # exactly the threshold set
        elif J.any():
            assert C.sum() == 1                         # one, the most confident
            i = int(np.flatnonzero(C)[0])
            assert conf[seg][i] == conf[seg][J].max()
            assert i == int(np.flatnonzero(J & (conf[seg] == conf[seg][J].max()))[0])
        assert committed[s] == C.sum()
        left = J & ~C
        assert int(new["active_block"][s]) == (a + 1 if not left.any() else a)


@pytest.mark.parametrize("seed", range(4))
def test_history_shift_only_where_masked(seed):
    st, conf = _random_state(100 + seed)
    nb = TR.num_blocks(st)
    new, _ = oracle.update_state(st, conf, nb, 0.9)
    m = st["masked"] == 1
    assert np.array_equal(new["conf2"][m], st["conf1"][m])
    assert np.array_equal(new["conf1"][m], conf[m])
    assert np.array_equal(new["hist_len"][m], np.minimum(st["hist_len"][m] + 1, 2))
    for k in ("conf1", "conf2", "hist_len"):
        assert np.array_equal(new[k][~m], st[k][~m])


def test_finished_sequence_is_untouched():
    st, conf = _random_state(7)
    nb = TR.num_blocks(st)
    st["active_block"][:] = nb + 1
    new, committed = oracle.update_state(st, conf, nb, 0.9)
    for k in st:
        assert np.array_equal(new[k], st[k])
    assert np.all(committed == 0)


def _params(cfg, **over):
    return {k: v for k, v in cfg.alloc_params(**over).items()}


@pytest.mark.parametrize("name", ["tiny_fp32", "llada_moe"])
def test_trajectory_terminates_within_bounds(name):
    cfg = W.CONFIGS[name]
    st = TR.initial_state(W.make_state(cfg, 0))
    ks, nfe, pairs, final = TC.oracle_trajectory(st, _params(cfg), seed=3)
    nb = TR.num_blocks(st)
    so = st["seq_offsets"]
    for s in range(nb.size):
        targets = int((st["block_id"][so[s]:so[s + 1]] > 0).sum())
        # at least one forward per block, at most one per target position
        assert nb[s] <= nfe[s] <= targets
    assert np.all(final["masked"] == 0)
    assert np.all(final["active_block"] == nb + 1)
    assert len(ks) == int(nfe.max())


def test_pairs_closed_form_under_fixed_counts():
    # uniform K_base (delta_role = delta_cur = 0): pairs of a sequence =
    # NFE x (positions per forward) x K_base, the paper's metric in closed form
    cfg = W.CONFIGS["tiny_fp32"]
    st = TR.initial_state(W.make_state(cfg, 1))
    ks, nfe, pairs, _ = TC.oracle_trajectory(st, _params(cfg, delta_role=0, delta_cur=0), seed=5)
    lens = np.diff(st["seq_offsets"])
    assert np.array_equal(pairs, nfe * lens * cfg.k_base)


def test_synthetic_confidence_is_deterministic_and_bounded():
    cfg = W.CONFIGS["llada_moe"]
    st = TR.initial_state(W.make_state(cfg, 0))
    ts = {k: torch.from_numpy(np.asarray(v)) for k, v in st.items()}
    sidx = torch.from_numpy(TR.seq_index(st))
    a = TR.synthetic_confidence(ts, 4, 11, sidx)
    b = TR.synthetic_confidence(ts, 4, 11, sidx)
    c = TR.synthetic_confidence(ts, 5, 11, sidx)
    assert torch.equal(a, b) and not torch.equal(a, c)
    assert float(a.min()) >= 0.0 and float(a.max()) <= 1.0
    # the 24-bit hash is close to uniform (chi-square over 64 bins)
    u = TR._uniform24(11, 3, torch.arange(1 << 16, dtype=torch.int64)).numpy()
    h = np.bincount((u * 64).astype(np.int64), minlength=64)
    e = u.size / 64
    assert ((h - e) ** 2 / e).sum() < 63 + 6 * np.sqrt(2 * 63)
