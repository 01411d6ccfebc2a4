"""Seeded random layer shapes through the whole forward, against the oracle.

Each case draws a shape (tokens, hidden size, experts, expert width, shared
expert, K bound), per-token counts and flags from its own seed, runs one
reflex_moe_forward and compares with the oracle's layer (Eq. 2 with the
TopK of the canonical scores): ids, offsets, permutation and row_of bit for
bit, alpha within ALPHA_RTOL, the output within the bf16 tolerance.  The
shapes cross the library's path choices (dense or screened or batched
scores, one-CTA or split dispatch, 1-SM or CTA-pair GEMMs, SIMT experts),
with ragged tails everywhere; the oracle's cost bounds the sizes.  The
weights have the benchmark layers' scale (std 0.02), where the outputs stay
below about 1 and the absolute bound is well above their bf16 rounding (at
std 0.05 the outputs of a 2048-wide layer reach about 12, whose bf16
half-ulp, 2^-5, is above the 2e-2 bound by itself).
"""
import numpy as np
import pytest

import gpu_cases as G
from paper_2608_01784_gb300 import _binding as B
from paper_2608_01784_gb300 import workloads as W

N_CASES = 48


def draw_case(seed: int) -> dict:
    rng = np.random.default_rng(10_000 + seed)
    E = int(rng.choice([1, 2, 3, 7, 8, 16, 31, 64, 65, 96, 128, 200, 256, 257, 512]))
    kmax = int(rng.integers(1, min(E, 16) + 1))
    d = int(rng.choice([128, 256, 384, 512, 640, 1024, 2048]))
    inter = int(rng.choice([64, 128, 192, 256, 320, 512]))
    shared = int(rng.choice([0, 0, 0, 64, 128, 256]))
    # token counts: mostly short, some past the batched-screen and split
    # dispatch thresholds (2048, 4096, 8192 tokens)
    band = rng.random()
    if band < 0.55:
        T = int(rng.integers(1, 1500))
    elif band < 0.85:
        T = int(rng.integers(2048, 5000))
    else:
        T = int(rng.integers(8192, 9000))
    # keep the oracle's expert work (T k d inter) to a few GFLOP
    while T * kmax * d * (inter + shared) > 3e9 and d > 128:
        d //= 2
        d -= d % 128
    kmode = str(rng.choice(["random", "max", "one", "skew"]))
    if kmode == "random":
        k = rng.integers(1, kmax + 1, T)
    elif kmode == "max":
        k = np.full(T, kmax)
    elif kmode == "one":
        k = np.ones(T)
    else:  # 70% at 1, 30% at k_max
        k = np.where(rng.random(T) < 0.7, 1, kmax)
    flags = 0 if rng.random() < 0.2 else B.REFLEX_FLAG_RENORM_TOPK
    if rng.random() < 0.15:
        flags |= B.REFLEX_FLAG_EXACT_SCORES
    if rng.random() < 0.15:
        flags |= B.REFLEX_FLAG_SIMT_EXPERTS
    return dict(T=T, d=d, E=E, inter=inter, shared=shared, kmax=kmax,
                k=k.astype(np.int32), flags=flags, seed=seed)


def test_draws_cover_the_paths():
    cases = [draw_case(s) for s in range(N_CASES)]
    assert any(c["T"] >= 8192 and c["E"] <= 64 for c in cases) or \
        any(c["T"] >= 2048 and 64 < c["E"] <= 256 for c in cases)
    assert any(c["shared"] for c in cases)
    assert any(c["flags"] & B.REFLEX_FLAG_SIMT_EXPERTS for c in cases)
    assert any(not c["flags"] & B.REFLEX_FLAG_RENORM_TOPK for c in cases)


@pytest.mark.gpu
@pytest.mark.parametrize("seed", range(N_CASES))
def test_random_layer_matches_the_oracle(seed):
    c = draw_case(seed)
    cfg = W.LayerConfig(name="fuzz", dtype="bf16", d=c["d"], E=c["E"], inter=c["inter"],
                        shared_inter=c["shared"], k_min=1, k_base=min(2, c["kmax"]),
                        k_max=c["kmax"], delta_role=1, delta_cur=1, w_cf=0.3, n_seq=1,
                        prompt_len=c["T"], gen_len=0, block=32, weight_std=0.02,
                        conf="uniform", mask_rule="half")
    layer = W.make_layer(cfg, 20_000 + seed, T=c["T"])
    gl = G.GpuLayer(cfg, layer)
    out, rec, status = gl.forward(c["k"], flags=c["flags"])
    shape = {key: c[key] for key in ("T", "d", "E", "inter", "shared", "kmax", "flags")}
    assert status == B.REFLEX_OK, shape
    renorm = bool(c["flags"] & B.REFLEX_FLAG_RENORM_TOPK)
    ref = G.oracle_layer(cfg, layer, c["k"], renorm=renorm)
    G.check_routing(rec, ref, c["k"], cfg.E)
    rel, mx = G.out_errors(out, ref["out"])
    assert rel <= G.BF16_REL_L2 and mx <= G.BF16_MAX_ABS, (shape, rel, mx)
