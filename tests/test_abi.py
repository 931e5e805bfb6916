"""The C-ABI library builds for sm_103a, loads, exports every entry point the
header declares, and rejects bad arguments on the host (no GPU needed: none
of these calls reaches the device)."""
import ctypes

import pytest

from paper_2608_07855_gb300 import build, commitkv as ck


@pytest.fixture(scope="module")
def lib():
    build.build()
    return ck.load_library()


def test_header_declares_the_entry_points():
    names = ck.declared_functions()
    for n in ("commitkv_page_effects", "commitkv_classify", "commitkv_joint_test", "commitkv_compact",
              "commitkv_compact_in_place", "commitkv_workspace_size", "commitkv_workspace_init", "commitkv_workspace_status",
              "commitkv_status_string"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for name in ck.declared_functions():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    for s in range(7):
        assert ck.status_string(s) and ck.status_string(s) != "unknown status"
    assert ck.status_string(99) == "unknown status"


def _good_traj(S=100, W=8, P=4, d=128, H=2):
    return ck.Traj(0x10000, 0x20000, H * S * d, S * d, d, 0x30000, S, 0x40000, 0x50000, W, 0x60000,
                   0x70000, P)


def test_workspace_size_host_only(lib):
    shape = ck.Shape(2, 2, 8, 128, ck.COMMITKV_BF16, 0.0)
    trajs = (ck.Traj * 1)(_good_traj())
    n = lib.commitkv_workspace_size(ctypes.byref(shape), 1, trajs)
    assert n > 256 and n % 256 == 0
    bad = ck.Shape(2, 3, 8, 128, ck.COMMITKV_BF16, 0.0)  # Hq not a multiple of H
    assert lib.commitkv_workspace_size(ctypes.byref(bad), 1, trajs) == 0
    assert lib.commitkv_workspace_size(ctypes.byref(shape), 0, trajs) == 0
    assert lib.commitkv_workspace_size(ctypes.byref(shape), 65, trajs) == 0


def test_host_validation(lib):
    shape = ck.Shape(2, 2, 8, 128, ck.COMMITKV_BF16, 0.0)
    trajs = (ck.Traj * 1)(_good_traj())
    R = (ctypes.c_void_p * 1)(0x80000)
    f = lib.commitkv_page_effects
    # unsupported head width
    s96 = ck.Shape(2, 2, 8, 96, ck.COMMITKV_BF16, 0.0)
    assert f(ctypes.byref(s96), 1, trajs, None, R, None, None, 0x90000, 1 << 30, None) == ck.COMMITKV_ERR_UNSUPPORTED
    # bad dtype, bad scale
    for bad in (ck.Shape(2, 2, 8, 128, 7, 0.0), ck.Shape(2, 2, 8, 128, 1, -1.0), ck.Shape(0, 2, 8, 128, 1, 0.0)):
        assert f(ctypes.byref(bad), 1, trajs, None, R, None, None, 0x90000, 1 << 30, None) == ck.COMMITKV_ERR_INVALID_ARG
    # missing outputs
    assert f(ctypes.byref(shape), 1, trajs, None, None, None, None, 0x90000, 1 << 30, None) == ck.COMMITKV_ERR_INVALID_ARG
    # missing / small / misaligned workspace
    assert f(ctypes.byref(shape), 1, trajs, None, R, None, None, None, 1 << 30, None) == ck.COMMITKV_ERR_WORKSPACE
    assert f(ctypes.byref(shape), 1, trajs, None, R, None, None, 0x90000, 1024, None) == ck.COMMITKV_ERR_WORKSPACE
    assert f(ctypes.byref(shape), 1, trajs, None, R, None, None, 0x90001, 1 << 30, None) == ck.COMMITKV_ERR_WORKSPACE
    # negative sizes, null pointers with work to do
    for kw in (dict(S=-1), dict(W=-1), dict(P=-1)):
        t = (ck.Traj * 1)(_good_traj(**{**dict(S=100, W=8, P=4), **kw}))
        assert f(ctypes.byref(shape), 1, t, None, R, None, None, 0x90000, 1 << 30, None) == ck.COMMITKV_ERR_INVALID_ARG
    t = _good_traj()
    t.k = None
    assert f(ctypes.byref(shape), 1, (ck.Traj * 1)(t), None, R, None, None, 0x90000, 1 << 30, None) == ck.COMMITKV_ERR_INVALID_ARG


def test_classify_and_compact_validation(lib):
    P = (ctypes.c_int32 * 1)(10)
    ptrs = (ctypes.c_void_p * 1)(0x1000)
    th = ck.Thresholds(0.01, 0.05, 0.75, 0.25)  # tau_dead > tau_use
    assert lib.commitkv_classify(1, P, ptrs, ptrs, ptrs, ctypes.byref(th), ptrs, ptrs, 0x2000, 0x90000, 1 << 20, None) \
        == ck.COMMITKV_ERR_INVALID_ARG
    th = ck.Thresholds(0.05, 0.01, 0.25, 0.75)  # rho_dead > rho_use
    assert lib.commitkv_classify(1, P, ptrs, ptrs, ptrs, ctypes.byref(th), ptrs, ptrs, 0x2000, 0x90000, 1 << 20, None) \
        == ck.COMMITKV_ERR_INVALID_ARG
    shape = ck.Shape(2, 2, 8, 128, ck.COMMITKV_BF16, 0.0)
    trajs = (ck.Traj * 1)(_good_traj())
    npend = (ctypes.c_int32 * 1)(0)
    # B_N > B
    assert lib.commitkv_compact(ctypes.byref(shape), 1, trajs, ptrs, None, npend, None, ptrs, 10, 11, 4,
                                ptrs, 0x3000, None, None, None, 0x90000, 1 << 20, None) == ck.COMMITKV_ERR_INVALID_ARG
    # too many pending pages
    npend = (ctypes.c_int32 * 1)(100000)
    assert lib.commitkv_compact(ctypes.byref(shape), 1, trajs, ptrs, ptrs, npend, ptrs, ptrs, 10, 5, 4,
                                ptrs, 0x3000, None, None, None, 0x90000, 1 << 20, None) == ck.COMMITKV_ERR_INVALID_ARG


def test_compact_in_place_validation(lib):
    """The in-place checkpoint checks its arguments like commitkv_compact and
    needs the cache's K, V and positions (it writes them)."""
    ptrs = (ctypes.c_void_p * 1)(0x1000)
    shape = ck.Shape(2, 2, 8, 128, ck.COMMITKV_BF16, 0.0)
    npend = (ctypes.c_int32 * 1)(0)
    trajs = (ck.Traj * 1)(_good_traj())
    # B_N > B
    assert lib.commitkv_compact_in_place(ctypes.byref(shape), 1, trajs, ptrs, None, npend, None, ptrs, 10, 11, 4,
                                         ptrs, 0x3000, 0x90000, 1 << 20, None) == ck.COMMITKV_ERR_INVALID_ARG
    # no K to compact
    bad = _good_traj()
    bad.k = None
    assert lib.commitkv_compact_in_place(ctypes.byref(shape), 1, (ck.Traj * 1)(bad), ptrs, None, npend, None, ptrs,
                                         10, 5, 4, ptrs, 0x3000, 0x90000, 1 << 20, None) == ck.COMMITKV_ERR_INVALID_ARG


def test_joint_and_variant_validation(lib):
    """Host checks of the joint test, the from-stats scoring and the
    classify variants: nothing is launched on a bad argument."""
    shape = ck.Shape(2, 2, 8, 128, ck.COMMITKV_BF16, 0.0)
    trajs = (ck.Traj * 1)(_good_traj())
    ptrs = (ctypes.c_void_p * 1)(0x1000)
    n_cand = 0x2000
    jt = lib.commitkv_joint_test
    # tau_joint NaN
    assert jt(ctypes.byref(shape), 1, trajs, None, ptrs, ptrs, n_cand, float("nan"), ptrs, None, 0x90000, 1 << 30,
              None) == ck.COMMITKV_ERR_INVALID_ARG
    # no stats / no candidates / no accepted output
    for st, cd, acc in ((None, ptrs, ptrs), (ptrs, None, ptrs), (ptrs, ptrs, None)):
        assert jt(ctypes.byref(shape), 1, trajs, None, st, cd, n_cand, 0.05, acc, None, 0x90000, 1 << 30,
                  None) == ck.COMMITKV_ERR_INVALID_ARG
    # workspace too small
    assert jt(ctypes.byref(shape), 1, trajs, None, ptrs, ptrs, n_cand, 0.05, ptrs, None, 0x90000, 4096,
              None) == ck.COMMITKV_ERR_WORKSPACE
    # the from-stats scoring needs its stats
    R = (ctypes.c_void_p * 1)(0x80000)
    assert lib.commitkv_page_effects_from_stats(ctypes.byref(shape), 1, trajs, None, None, R, None, 0x90000, 1 << 30,
                                                None) == ck.COMMITKV_ERR_INVALID_ARG
    # classify variants: unknown bits
    P = (ctypes.c_int32 * 1)(10)
    th = ck.Thresholds(0.05, 0.01, 0.75, 0.25)
    cv = lib.commitkv_classify_variant
    assert cv(1, P, ptrs, ptrs, ptrs, ctypes.byref(th), 4, ptrs, ptrs, 0x2000, 0x90000, 1 << 20,
              None) == ck.COMMITKV_ERR_INVALID_ARG
    # a negative page count
    Pn = (ctypes.c_int32 * 1)(-1)
    assert cv(1, Pn, ptrs, ptrs, ptrs, ctypes.byref(th), 0, ptrs, ptrs, 0x2000, 0x90000, 1 << 20,
              None) == ck.COMMITKV_ERR_INVALID_ARG


def test_workspace_covers_smaller_caches(lib):
    """A workspace sized for the post-commit caches serves the pre-commit
    call too (its S and P are smaller), for every chunking regime."""
    for dtype, d in ((ck.COMMITKV_BF16, 128), (ck.COMMITKV_F32, 64), (ck.COMMITKV_BF16, 64)):
        shape = ck.Shape(4, 8, 32, d, dtype, 0.0)
        for S_post in (300, 1500, 16384 + 2080, 36896, 139328):
            big = lib.commitkv_workspace_size(ctypes.byref(shape), 1, (ck.Traj * 1)(_good_traj(S=S_post, W=32, P=S_post // 40, d=d, H=8)))
            for S in range(max(1, S_post - 5000), S_post + 1, 97):
                small = lib.commitkv_workspace_size(ctypes.byref(shape), 1, (ck.Traj * 1)(_good_traj(S=S, W=32, P=S // 40, d=d, H=8)))
                assert 0 < small <= big, (d, S_post, S, small, big)
