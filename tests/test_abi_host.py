"""Host-side checks of the C ABI (no GPU needed): the library builds for
sm_103a, exports every entry point include/reflex.h declares, and rejects bad
arguments before anything is enqueued."""
import ctypes
import re
import shutil
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]
HEADER = ROOT / "include" / "reflex.h"

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and
                                not Path("/usr/local/cuda/bin/nvcc").exists(),
                                reason="needs nvcc to build the library")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_01784_gb300 import build, _binding
    build.build()
    return _binding.load()


def declared_functions():
    text = HEADER.read_text()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(reflex_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("reflex_allocate", "reflex_moe_forward",
                 "reflex_moe_workspace_size", "reflex_moe_status"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2608_01784_gb300 import _binding
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert name in _binding.EXPORTED, name


def test_status_strings_and_version(lib):
    from paper_2608_01784_gb300 import _binding as B
    assert B.reflex_status_string(B.REFLEX_OK) == "ok"
    assert "workspace" in B.reflex_status_string(B.REFLEX_EWORKSPACE)
    assert B.reflex_status_string(999) == "unknown status"
    assert B.reflex_abi_version() == B.ABI_VERSION == 114


def test_default_params_are_the_paper_settings(lib):
    from paper_2608_01784_gb300 import _binding as B
    p = B.reflex_default_params()
    assert (p.k_base, p.delta_role, p.delta_cur) == (8, 4, 2)
    assert p.q == pytest.approx(0.25) and p.theta == pytest.approx(0.9)
    assert p.v_ref == pytest.approx(0.01) and p.tau == pytest.approx(0.05)
    assert p.w_cf == pytest.approx(0.30)
    # the ablation fields sit where the C struct has them (a layout mismatch
    # would show up as garbage here): FPS, no shuffle
    assert (p.signal, p.role_shuffle, p.shuffle_seed) == (B.REFLEX_SIGNAL_FPS, 0, 0)
    assert (p.count_rule, p.rule_threshold) == (B.REFLEX_RULE_REFLEX, 0.0)
    assert ctypes.sizeof(B.reflex_alloc_params) == 64


def test_workspace_size(lib):
    from paper_2608_01784_gb300 import _binding as B
    ws = B.reflex_moe_workspace_size
    a = ws(1, 1024, 2048, 64, 1024, 0, 12)
    assert a > 1024 * 12 * 2048 * 2          # at least the gathered rows
    assert ws(1, 2048, 2048, 64, 1024, 0, 12) > a
    assert ws(1, 1024, 2048, 64, 1024, 512, 12) > a   # shared expert buffers
    assert ws(0, 1024, 2048, 64, 1024, 0, 12) > a     # fp32 storage
    assert ws(1, 1024, 2000, 64, 1024, 0, 12) == 0    # d % 64
    assert ws(1, 1024, 2048, 0, 1024, 0, 12) == 0     # E >= 1
    assert ws(1, 1024, 2048, 64, 1024, 0, 33) == 0    # k_max <= 32
    assert ws(7, 1024, 2048, 64, 1024, 0, 12) == 0    # dtype


def test_workspace_size_never_shrinks_with_more_tokens(lib):
    # a workspace sized for a batch serves every smaller one (MoELayer sizes
    # it once for max_tokens), across the switch from 32- to 256-token
    # dispatch blocks at 4096 tokens and the router-screen regions
    from paper_2608_01784_gb300 import _binding as B
    ws = B.reflex_moe_workspace_size
    # every T up to 12000 (the score region's split count falls at 128-row
    # tile boundaries such as 512 -> 513 tokens with 256 experts), then a
    # sample up to 65536
    Ts = list(range(0, 12001)) + list(range(12001, 65537, 997)) + [65536]
    for dtype, d, E, inter, shared in [(1, 2048, 64, 1024, 0), (1, 2048, 256, 512, 512),
                                       (1, 2048, 128, 1024, 0), (0, 256, 8, 128, 0),
                                       (1, 512, 160, 256, 0)]:
        prev = 0
        for T in Ts:
            cur = ws(dtype, T, d, E, inter, shared, 12)
            assert cur >= prev, (dtype, d, E, T, prev, cur)
            prev = cur


def test_host_rejections_enqueue_nothing(lib):
    from paper_2608_01784_gb300 import _binding as B
    p = B.reflex_default_params()
    # null parameter block / bad parameters
    assert lib.reflex_allocate(None, None, None, None, None, None, None, None,
                               4, 1, 8, None, None, None, None, None) == B.REFLEX_EINVAL
    bad = B.make_params(q=0.7)
    assert lib.reflex_allocate(None, 1, 1, 1, 1, 1, 1, 1, 4, 1, 8,
                               ctypes.byref(bad), 1, None, None, None) == B.REFLEX_EINVAL
    bad = B.make_params(k_min=5, k_max=4)
    assert lib.reflex_allocate(None, 1, 1, 1, 1, 1, 1, 1, 4, 1, 8,
                               ctypes.byref(bad), 1, None, None, None) == B.REFLEX_EINVAL
    for bad in (B.make_params(signal=5), B.make_params(signal=-1),
                B.make_params(role_shuffle=2)):
        assert lib.reflex_allocate(None, 1, 1, 1, 1, 1, 1, 1, 4, 1, 8,
                                   ctypes.byref(bad), 1, None, None, None) == B.REFLEX_EINVAL
    assert lib.reflex_allocate(None, 1, 1, 1, 1, 1, 1, 1, 4, 0, 8,
                               ctypes.byref(p), 1, None, None, None) == B.REFLEX_EINVAL
    # forward: bad shapes, missing workspace
    fw = lib.reflex_moe_forward
    assert fw(1, 1, 1, 1, 1, None, None, 0, 1, 4, 2000, 8, 128, 4, 1, 1, 1 << 30,
              1, None, None) == B.REFLEX_EINVAL
    assert fw(1, 1, 1, 1, 1, None, None, 0, 1, 4, 256, 8, 128, 4, 1, None, 0,
              1, None, None) == B.REFLEX_EWORKSPACE
    need = B.reflex_moe_workspace_size(1, 4, 256, 8, 128, 0, 4)
    assert fw(1, 1, 1, 1, 1, None, None, 0, 1, 4, 256, 8, 128, 4, 1, 256,
              need - 1, 1, None, None) == B.REFLEX_EWORKSPACE
    # misaligned workspace
    assert fw(1, 1, 1, 1, 1, None, None, 0, 1, 4, 256, 8, 128, 4, 1, 257,
              need, 1, None, None) == B.REFLEX_EWORKSPACE
    # shared expert declared without weights
    assert fw(1, 1, 1, 1, 1, None, None, 128, 1, 4, 256, 8, 128, 4, 1, 256,
              1 << 30, 1, None, None) == B.REFLEX_EINVAL
    # T = 0 launches no kernel; it fills the record and clears the workspace
    # header with a memset, which needs a device (none here: ECUDA)
    rec = B.reflex_route_record()
    assert fw(1, None, None, None, None, None, None, 0, None, 0, 256, 8, 128, 4,
              1, 256, 1 << 20, None, ctypes.byref(rec), None) == B.REFLEX_ECUDA
    assert rec.ids == 3 * 256            # after the header, scores and expert norms
    assert lib.reflex_selftest_wait_timeout(None, 10, None) == B.REFLEX_EINVAL
    assert lib.reflex_read_status(None, None) == B.REFLEX_EINVAL


def test_update_state_host_rejections(lib):
    from paper_2608_01784_gb300 import _binding as B
    # every check returns before a pointer is used
    assert lib.reflex_update_state(None, None, None, None, None, None, None, None, None,
                                   4, 0, 0.9, None, None, None) == B.REFLEX_EINVAL
    assert lib.reflex_update_state(None, None, None, None, None, None, 1, 1, 1,
                                   4, 1, 0.9, None, None, None) == B.REFLEX_EINVAL
    assert lib.reflex_update_state(1, 1, 1, 1, 1, 1, 1, 1, 1, 4, 1, float("nan"),
                                   None, None, None) == B.REFLEX_EINVAL


def test_step_host_rejections(lib):
    # reflex_step checks both halves before it launches anything
    import ctypes
    from paper_2608_01784_gb300 import _binding as B
    p = B.reflex_alloc_params()
    lib.reflex_default_params(ctypes.byref(p))
    state = (1, 1, 1, 1, 1, 1, 1)          # dummy device pointers, never read

    def step(B_=1, params=ctypes.byref(p), T=4, d=256, ws=1 << 30, k_out=1, q=None):
        return lib.reflex_step(*state, B_, params, k_out, None, None, 1, 1, 1, 1, 1,
                               None, None, 0, T, d, 8, 128, 4, 1, 256, ws, 1, None, None)
    assert step(params=None) == B.REFLEX_EINVAL          # no allocation parameters
    assert step(B_=0) == B.REFLEX_EINVAL                 # no sequence
    assert step(k_out=None) == B.REFLEX_EINVAL           # nowhere to put the counts
    assert step(d=100) == B.REFLEX_EINVAL                # forward shape rule
    assert step(ws=16) == B.REFLEX_EWORKSPACE            # workspace too small
    bad = B.reflex_alloc_params()
    lib.reflex_default_params(ctypes.byref(bad))
    bad.q = 0.75                                         # q outside (0, 1/2]
    assert step(params=ctypes.byref(bad)) == B.REFLEX_EINVAL


def test_step_launch_counts_of_the_bench_layers():
    # the kernels of one reflex_step as the ncu launch lists show them:
    # LLaDA-MoE layer (count, scores, selection, count + scan, gather, two
    # GEMMs, combine), LLaDA2.0-mini layer (count, norms, score GEMM,
    # screened selection, count, scan, gather, four GEMMs, combine), 32 x 1024
    # layer (count, norms, score GEMM, batched recheck, count, scan, gather,
    # two GEMMs, combine)
    from paper_2608_01784_gb300 import _binding as B
    from paper_2608_01784_gb300 import api
    assert api.step_launches("bf16", 1024, 2048, 64, 0) == 8
    assert api.step_launches("bf16", 8192, 2048, 256, 512) == 12
    assert api.step_launches("bf16", 32768, 2048, 64, 0) == 10   # batched screen
    assert api.step_launches("bf16", 4096, 2048, 64, 0) == 8      # dense scores
    # exact scores: the screen's three kernels become scores + selection
    exact = B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_FLAG_EXACT_SCORES
    assert api.step_launches("bf16", 8192, 2048, 256, 512, flags=exact) == 11


def test_count_rule_host_rejections(lib):
    # the score rules: every check returns before anything is launched
    import ctypes
    from paper_2608_01784_gb300 import _binding as B
    for rule, thr in ((3, 0.2), (-1, 0.2), (B.REFLEX_RULE_TOP_P, float("nan")),
                      (B.REFLEX_RULE_EXPERT_THRESHOLD, float("inf"))):
        p = B.make_params(count_rule=rule, rule_threshold=thr)
        assert lib.reflex_allocate(1, None, None, None, None, None, None, None, 4, 1, 8,
                                   ctypes.byref(p), 1, None, None, None) == B.REFLEX_EINVAL
    p = B.make_params(count_rule=B.REFLEX_RULE_TOP_P, rule_threshold=0.2)
    # no score matrix, or an expert count outside [1, 1024]
    assert lib.reflex_allocate(None, None, None, None, None, None, None, None, 4, 1, 8,
                               ctypes.byref(p), 1, None, None, None) == B.REFLEX_EINVAL
    for E in (0, 1025):
        assert lib.reflex_allocate(1, None, None, None, None, None, None, None, 4, 1, E,
                                   ctypes.byref(p), 1, None, None, None) == B.REFLEX_EINVAL
    # nowhere to put the counts
    assert lib.reflex_allocate(1, None, None, None, None, None, None, None, 4, 1, 8,
                               ctypes.byref(p), None, None, None, None) == B.REFLEX_EINVAL

    # reflex_step: the counts come out of the ROUTE stage, so a stage subset
    # without it is rejected
    def step(flags):
        return lib.reflex_step(None, None, None, None, None, None, None, 1, ctypes.byref(p),
                               1, None, None, 1, 1, 1, 1, 1, None, None, 0, 4, 256, 8, 128,
                               4, flags, 256, 1 << 30, 1, None, None)
    assert step(B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_STAGE_DISPATCH) == B.REFLEX_EINVAL
    assert step(B.REFLEX_STAGE_EXPERT_UP | B.REFLEX_STAGE_COMBINE) == B.REFLEX_EINVAL


def test_default_params_count_rule_is_reflex(lib):
    import ctypes
    from paper_2608_01784_gb300 import _binding as B
    p = B.reflex_alloc_params()
    p.count_rule, p.rule_threshold = 9, 9.0
    lib.reflex_default_params(ctypes.byref(p))
    assert p.count_rule == B.REFLEX_RULE_REFLEX and p.rule_threshold == 0.0
    assert ctypes.sizeof(B.reflex_alloc_params) == 64
