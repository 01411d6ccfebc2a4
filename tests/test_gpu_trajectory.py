"""GPU parity of the refinement-state update (Sec. 3.1, Eq. 1) and of whole
denoising trajectories: the CUDA path through the C ABI against the oracle on
the same states and the same (exact, device-independent) synthetic
confidences.  Every state array, every per-forward count vector, NFE and pairs
must match bit for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_01784_gb300 import _binding as B
from paper_2608_01784_gb300 import api
from paper_2608_01784_gb300 import trajectory as TR
from paper_2608_01784_gb300 import workloads as W
from tests import trajectory_cases as TC

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_01784_gb300 import build
    build.build()
    B.load()
    oracle.build()


def _gpu_update(st: dict, conf: np.ndarray, nb: np.ndarray, theta: float):
    ds = api.state_to_device(st)
    committed = torch.zeros(nb.size, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    api.update_state(ds, torch.from_numpy(conf).cuda(), torch.from_numpy(nb).cuda(), theta,
                     committed=committed, status=status)
    torch.cuda.synchronize()
    return ({k: v.cpu().numpy() for k, v in ds.items()}, committed.cpu().numpy(),
            B.reflex_read_status(status))


@pytest.mark.parametrize("name", ["tiny_fp32", "llada_moe", "llada2_mini", "llada_moe_b32"])
@pytest.mark.parametrize("seed", range(3))
@pytest.mark.parametrize("theta", [0.9, 0.7, 1.01])
def test_update_state_bit_exact(name, seed, theta):
    cfg = W.CONFIGS[name]
    st = W.make_state(cfg, seed, hist_len=None)
    rng = np.random.default_rng(seed)
    st["hist_len"] = rng.integers(0, 3, st["hist_len"].size).astype(np.uint8)
    conf = rng.uniform(0.0, 1.0, st["block_id"].size).astype(np.float32)
    conf[rng.integers(0, conf.size, 64)] = 0.5      # ties for the fallback
    nb = TR.num_blocks(st)
    st["active_block"][0] = nb[0] + 1               # one finished sequence
    gpu, c_gpu, status = _gpu_update(st, conf, nb, theta)
    ref, c_ref = oracle.update_state(st, conf, nb, theta)
    assert status == B.REFLEX_OK
    for k in ("masked", "conf1", "conf2", "hist_len", "active_block"):
        assert np.array_equal(gpu[k], ref[k]), k
    assert np.array_equal(c_gpu, c_ref)


def test_update_state_golden():
    import json, os
    gold = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                       "trajectory_worked.json")))
    bid = np.array(gold["block_id"], np.int32)
    T = bid.size
    st = dict(conf1=np.zeros(T, np.float32), conf2=np.zeros(T, np.float32),
              hist_len=np.zeros(T, np.uint8), masked=(bid > 0).astype(np.uint8),
              block_id=bid, seq_offsets=np.array([0, T], np.int32),
              active_block=np.array([1], np.int32))
    nb = np.array([gold["num_blocks"]], np.int32)
    for f in gold["forwards"]:
        st, committed, status = _gpu_update(st, np.array(f["conf"], np.float32), nb,
                                            gold["theta"])
        assert status == B.REFLEX_OK
        assert st["masked"].tolist() == f["masked_after"], f["why"]
        assert int(st["active_block"][0]) == f["active_after"], f["why"]
        assert int(committed[0]) == f["committed"], f["why"]


@pytest.mark.parametrize("name,variant", [
    ("tiny_fp32", {}), ("llada_moe", {}), ("llada_moe", dict(delta_role=0, delta_cur=0)),
    ("llada2_mini", {}), ("llada2_mini", dict(signal=B.REFLEX_SIGNAL_PROGRESS)),
])
def test_trajectory_matches_oracle(name, variant):
    cfg = W.CONFIGS[name]
    st = TR.initial_state(W.make_state(cfg, 2))
    params = cfg.alloc_params(**variant)
    ks_ref, nfe_ref, pairs_ref, final_ref = TC.oracle_trajectory(st, params, seed=9)
    ds = api.state_to_device(st)
    record = []
    res = TR.simulate(ds, B.make_params(**params), cfg.E, seed=9, record=record)
    assert res["alloc_status"] == B.REFLEX_OK and res["update_status"] == B.REFLEX_OK
    assert res["forwards"] == len(ks_ref)
    for t, (kg, kr) in enumerate(zip(record, ks_ref)):
        assert np.array_equal(kg.cpu().numpy(), kr), f"forward {t}"
    assert np.array_equal(res["nfe"], nfe_ref)
    assert np.array_equal(res["pairs"], pairs_ref)
    for k in ("masked", "active_block", "conf1", "conf2", "hist_len"):
        assert np.array_equal(ds[k].cpu().numpy(), final_ref[k]), k


def test_trajectory_with_layer_runs_clean():
    # the same loop with the MoE layer in every forward: statuses stay clean
    # and the counts are those of the layer-free run
    cfg = W.CONFIGS["llada_moe"]
    st = TR.initial_state(W.make_state(cfg, 4))
    layer = W.make_layer(cfg, 4)
    dl = api.layer_to_device(layer, cfg.dtype)
    moe = api.MoELayer(dl, dtype=cfg.dtype, d=cfg.d, E=cfg.E, inter=cfg.inter,
                       shared_inter=cfg.shared_inter, k_max=cfg.k_max, max_tokens=cfg.T)
    p = B.make_params(**cfg.alloc_params())
    r1 = TR.simulate(api.state_to_device(st), p, cfg.E, seed=1, moe=moe, hidden=dl["hidden"])
    r2 = TR.simulate(api.state_to_device(st), p, cfg.E, seed=1)
    assert moe.status() == B.REFLEX_OK
    assert np.array_equal(r1["nfe"], r2["nfe"]) and np.array_equal(r1["pairs"], r2["pairs"])


def test_trajectory_graph_replay_matches_eager():
    cfg = W.CONFIGS["llada2_mini"]
    st = TR.initial_state(W.make_state(cfg, 6))
    p = B.make_params(**cfg.alloc_params())
    ds_e, ds_g = api.state_to_device(st), api.state_to_device(st)
    r_e = TR.simulate(ds_e, p, cfg.E, seed=2)
    r_g = TR.simulate(ds_g, p, cfg.E, seed=2, graph=True, check_every=8)
    assert np.array_equal(r_e["nfe"], r_g["nfe"])
    assert np.array_equal(r_e["pairs"], r_g["pairs"])
    assert r_g["alloc_status"] == B.REFLEX_OK and r_g["update_status"] == B.REFLEX_OK
    for k in ("masked", "active_block", "conf1", "conf2", "hist_len"):
        assert torch.equal(ds_e[k], ds_g[k]), k

