"""The routing entry point that allocates nothing (reflex_route_noalloc).

It exists for callers that cannot obtain device memory of their own (a host
framework owns the allocator, a plugin may only use the buffers it is given,
or cudaMalloc is not allowed after start-up): its score scratch lives in a
fixed array inside the library.  Its results must equal the oracle's routing
(selected experts bit for bit, weights within the routing tolerance) and the
routing record of the regular workspace-based forward, call after call, even
though every call reuses the same array.  This file is collected last on
purpose.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_01784_gb300 import _binding as B
from paper_2608_01784_gb300 import workloads as W
from tests import gpu_cases as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_01784_gb300 import build
    build.build()
    B.load()


def _noalloc(dtype, hidden, w_router, k, T, d, E, k_max, flags=B.REFLEX_FLAG_RENORM_TOPK):
    kd = torch.from_numpy(np.ascontiguousarray(k, np.int32)).cuda()
    ids = torch.full((T, k_max), -7, dtype=torch.int32, device="cuda")
    alpha = torch.full((T, k_max), -7.0, dtype=torch.float32, device="cuda")
    st = torch.full((1,), 123, dtype=torch.int32, device="cuda")   # stale value
    rc = B.reflex_route_noalloc(dtype, hidden, w_router, kd, T, d, E, k_max, flags,
                                ids, alpha, st)
    assert rc == B.REFLEX_OK
    assert B.reflex_read_status(st) == B.REFLEX_OK
    return ids.cpu().numpy(), alpha.cpu().numpy()


def _oracle_routing(hidden_host, w_router_host, k, k_max, renorm=True):
    z = oracle.router_logits(hidden_host, w_router_host)
    return oracle.select(z, k, k_max, renorm)


def _check_vs_oracle(ids, alpha, ref):
    ids_ref, alpha_ref = ref
    assert np.array_equal(ids, ids_ref), "selected experts differ from the oracle"
    valid = ids_ref >= 0
    np.testing.assert_allclose(alpha[valid], alpha_ref[valid], rtol=G.ALPHA_RTOL, atol=1e-7)
    assert np.all(alpha[~valid] == 0)


def _route_both(cfg, layer, k):
    gl = G.GpuLayer(cfg, layer)
    _, rec, status = gl.forward(k)
    assert status == B.REFLEX_OK
    dtype = B.REFLEX_DTYPE_BF16 if cfg.dtype == "bf16" else B.REFLEX_DTYPE_F32
    ids, alpha = _noalloc(dtype, gl.dev["hidden"], gl.dev["w_router"], k, cfg.T, cfg.d,
                          cfg.E, cfg.k_max)
    return rec, ids, alpha


def test_noalloc_routing_matches_oracle_and_forward_on_consecutive_calls():
    # calls in a row on different inputs: the shared scratch array holds the
    # previous call's scores when the next one starts
    for name, seed in (("llada_moe", 0), ("tiny_fp32", 1), ("llada_moe", 2)):
        cfg = W.CONFIGS[name]
        layer = W.make_layer(cfg, seed)
        k = G.oracle_allocate(W.make_state(cfg, seed), G.params_of(cfg))
        rec, ids, alpha = _route_both(cfg, layer, k)
        _check_vs_oracle(ids, alpha, _oracle_routing(layer["hidden"], layer["w_router"], k,
                                                     cfg.k_max))
        assert np.array_equal(ids, rec["ids"])
        valid = rec["ids"] >= 0
        np.testing.assert_allclose(alpha[valid], rec["alpha"][valid],
                                   rtol=G.ALPHA_RTOL, atol=1e-7)


def test_noalloc_at_the_scratch_limit_bf16_256_experts():
    # T * E = 4096 x 256 = the array's size exactly.  The workspace forward
    # screens these scores with the tensor-core GEMM while the no-alloc call
    # computes every score with the chain: two different paths, same bits.
    cfg = W.CONFIGS["llada2_mini"]
    T, E, d = 4096, cfg.E, cfg.d
    assert T * E == B.REFLEX_NOALLOC_MAX_SCORES
    hidden = W.make_hidden(cfg, 11, T)
    w_router = W.to_bf16_bits(W.normal_f32(11, "noalloc/w_router", E * d, 0.02)).reshape(E, d)
    k = G.oracle_allocate(W.make_state(cfg, 11, T=T), G.params_of(cfg))
    assert k.size == T
    hd = torch.from_numpy(hidden.view(np.int16)).cuda().view(torch.bfloat16)
    wd = torch.from_numpy(w_router.view(np.int16)).cuda().view(torch.bfloat16)
    ref = _oracle_routing(hidden, w_router, k, cfg.k_max)
    for _ in range(2):   # two calls in a row on the same full array
        ids, alpha = _noalloc(B.REFLEX_DTYPE_BF16, hd, wd, k, T, d, E, cfg.k_max)
        _check_vs_oracle(ids, alpha, ref)
    # the workspace forward's screened routing agrees
    from paper_2608_01784_gb300 import api
    moe = api.MoELayer(dict(w_router=wd, w_gate_up=wd, w_down=wd), dtype="bf16", d=d, E=E,
                       inter=cfg.inter, shared_inter=0, k_max=cfg.k_max, max_tokens=T)
    kd = torch.from_numpy(k).cuda()
    out = torch.empty((T, d), dtype=torch.bfloat16, device="cuda")
    moe.forward(hd, kd, out, B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_ROUTE)
    torch.cuda.synchronize()
    assert moe.status() == B.REFLEX_OK
    assert np.array_equal(moe.record()["ids"].cpu().numpy(), ids)


def test_noalloc_rejects_too_many_scores():
    for T, E in ((8192, 256), (4097, 256), (1 + (1 << 20) // 64, 64)):
        assert T * E > B.REFLEX_NOALLOC_MAX_SCORES
        rc = B.reflex_route_noalloc(B.REFLEX_DTYPE_BF16, 1, 1, 1, T, 2048, E, 12,
                                    B.REFLEX_FLAG_RENORM_TOPK, 1, 1)
        assert rc == B.REFLEX_EWORKSPACE


def test_noalloc_zero_tokens_clears_a_stale_status():
    st = torch.full((1,), 5, dtype=torch.int32, device="cuda")
    rc = B.reflex_route_noalloc(B.REFLEX_DTYPE_BF16, None, None, None, 0, 2048, 64, 12,
                                B.REFLEX_FLAG_RENORM_TOPK, None, None, st)
    assert rc == B.REFLEX_OK
    assert B.reflex_read_status(st) == B.REFLEX_OK
