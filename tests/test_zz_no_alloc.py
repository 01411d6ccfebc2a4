"""The routing entry point that allocates nothing (reflex_route_noalloc).

It exists for callers that cannot obtain device memory of their own (a host
framework owns the allocator, a plugin may only use the buffers it is given,
or cudaMalloc is not allowed after start-up): its score scratch lives in a
fixed array inside the library.  Its results must equal the routing record of
the regular workspace-based forward, call after call, even though every call
reuses the same array.  This file is collected last on purpose.
"""
import numpy as np
import pytest
import torch

from paper_2608_01784_gb300 import _binding as B
from paper_2608_01784_gb300 import workloads as W
from tests import gpu_cases as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_01784_gb300 import build
    build.build()
    B.load()


def _route_both(cfg, layer, k):
    gl = G.GpuLayer(cfg, layer)
    _, rec, status = gl.forward(k)
    assert status == B.REFLEX_OK
    T = cfg.T
    kd = torch.from_numpy(np.ascontiguousarray(k, np.int32)).cuda()
    ids = torch.full((T, cfg.k_max), -7, dtype=torch.int32, device="cuda")
    alpha = torch.full((T, cfg.k_max), -7.0, dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    dtype = B.REFLEX_DTYPE_BF16 if cfg.dtype == "bf16" else B.REFLEX_DTYPE_F32
    rc = B.reflex_route_noalloc(dtype, gl.dev["hidden"], gl.dev["w_router"], kd,
                                T, cfg.d, cfg.E, cfg.k_max,
                                B.REFLEX_FLAG_RENORM_TOPK, ids, alpha, st)
    assert rc == B.REFLEX_OK
    assert B.reflex_read_status(st) == B.REFLEX_OK
    return rec, ids.cpu().numpy(), alpha.cpu().numpy()


def test_noalloc_routing_matches_forward_on_consecutive_calls():
    # two calls in a row on different inputs: the shared scratch array holds
    # the first call's scores when the second one starts
    for name, seed in (("llada_moe", 0), ("tiny_fp32", 1), ("llada_moe", 2)):
        cfg = W.CONFIGS[name]
        layer = W.make_layer(cfg, seed)
        k = G.oracle_allocate(W.make_state(cfg, seed), G.params_of(cfg))
        rec, ids, alpha = _route_both(cfg, layer, k)
        assert np.array_equal(ids, rec["ids"])
        valid = rec["ids"] >= 0
        np.testing.assert_allclose(alpha[valid], rec["alpha"][valid],
                                   rtol=G.ALPHA_RTOL, atol=1e-7)
        assert np.all(alpha[~valid] == 0)


def test_noalloc_rejects_too_many_scores():
    T, E = 8192, 256            # T * E = 2^21 > the fixed array
    assert T * E > B.REFLEX_NOALLOC_MAX_SCORES
    rc = B.reflex_route_noalloc(B.REFLEX_DTYPE_BF16, 1, 1, 1, T, 2048, E, 12,
                                B.REFLEX_FLAG_RENORM_TOPK, 1, 1)
    assert rc == B.REFLEX_EWORKSPACE
