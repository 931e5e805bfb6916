"""Python binding of the CommitKV C ABI (include/commitkv.h).

Argument marshalling only: every step of the hot path runs in the CUDA
kernels of libcommitkv.so.  Tensors are torch tensors on the GPU (torch is
used for device memory and streams); the functions carry the C names.
There is no CPU fallback: without the compiled library or a GPU every call
raises.
"""
from __future__ import annotations

import ctypes
import os
import re
from dataclasses import dataclass
from typing import Optional, Sequence

from . import build as _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "commitkv.h")
HEADERS = [os.path.join(ROOT, "include", f) for f in ("commitkv.h", "commitkv_testing.h")]

COMMITKV_OK = 0
COMMITKV_ERR_INVALID_ARG = 1
COMMITKV_ERR_UNSUPPORTED = 2
COMMITKV_ERR_CUDA = 3
COMMITKV_ERR_TIMEOUT = 4
COMMITKV_ERR_WORKSPACE = 5
COMMITKV_ERR_DEVICE_INPUT = 6
COMMITKV_F32 = 0
COMMITKV_BF16 = 1
MAX_TRAJ = 64


class CommitKVError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


class Shape(ctypes.Structure):
    _fields_ = [("layers", ctypes.c_int32), ("kv_heads", ctypes.c_int32),
                ("q_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("softmax_scale", ctypes.c_float)]


class Traj(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("stride_layer", ctypes.c_int64), ("stride_head", ctypes.c_int64),
                ("stride_tok", ctypes.c_int64), ("pos", ctypes.c_void_p), ("S", ctypes.c_int32),
                ("q", ctypes.c_void_p), ("q_pos", ctypes.c_void_p), ("W", ctypes.c_int32),
                ("page_start", ctypes.c_void_p), ("page_len", ctypes.c_void_p),
                ("P", ctypes.c_int32)]


class Thresholds(ctypes.Structure):
    _fields_ = [("tau_use", ctypes.c_float), ("tau_dead", ctypes.c_float),
                ("rho_use", ctypes.c_float), ("rho_dead", ctypes.c_float)]


_lib = None


def library_path() -> str:
    return _build.LIB


def load_library(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libcommitkv.so (building it in-tree with nvcc if needed)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path) or not _build.up_to_date():
        if not build_if_missing:
            raise RuntimeError(f"CommitKV CUDA library missing: {path}")
        path = _build.build()
    lib = ctypes.CDLL(path)
    vp, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    P = ctypes.POINTER
    lib.commitkv_workspace_size.argtypes = [P(Shape), i32, P(Traj)]
    lib.commitkv_workspace_size.restype = sz
    lib.commitkv_workspace_init.argtypes = [vp, sz, vp]
    lib.commitkv_workspace_status.argtypes = [vp, sz, vp, i32]
    lib.commitkv_status_string.argtypes = [ctypes.c_int]
    lib.commitkv_status_string.restype = ctypes.c_char_p
    lib.commitkv_page_effects.argtypes = [P(Shape), i32, P(Traj), vp, vp, vp, vp, vp, sz, vp]
    lib.commitkv_page_effects_from_stats.argtypes = [P(Shape), i32, P(Traj), vp, vp, vp, vp, vp, sz, vp]
    lib.commitkv_classify.argtypes = [i32, vp, vp, vp, vp, P(Thresholds), vp, vp, vp, vp, sz, vp]
    lib.commitkv_classify_variant.argtypes = [i32, vp, vp, vp, vp, P(Thresholds), ctypes.c_uint32, vp, vp, vp,
                                              vp, sz, vp]
    lib.commitkv_joint_test.argtypes = [P(Shape), i32, P(Traj), vp, vp, vp, vp, ctypes.c_float,
                                        vp, vp, vp, sz, vp]
    lib.commitkv_compact.argtypes = [P(Shape), i32, P(Traj), vp, vp, vp, vp, vp, i32, i32, i32,
                                     vp, vp, vp, vp, vp, vp, sz, vp]
    lib.commitkv_compact_in_place.argtypes = [P(Shape), i32, P(Traj), vp, vp, vp, vp, vp, i32, i32, i32,
                                              vp, vp, vp, sz, vp]
    lib.commitkv_compact_noalloc.argtypes = [P(Shape), i32, P(Traj), vp, vp, vp, vp, vp, i32, i32,
                                             i32, vp, vp, vp, vp, vp, vp, vp]
    lib.commitkv_test_barrier_timeout.argtypes = [vp, sz, i32, vp]
    lib.commitkv_token_scores.argtypes = [P(Shape), i32, P(Traj), vp, vp, vp, vp, sz, vp]
    for f in ("commitkv_workspace_init", "commitkv_workspace_status", "commitkv_page_effects",
              "commitkv_page_effects_from_stats", "commitkv_classify", "commitkv_classify_variant",
              "commitkv_joint_test", "commitkv_compact", "commitkv_compact_in_place", "commitkv_compact_noalloc",
              "commitkv_test_barrier_timeout", "commitkv_token_scores"):
        getattr(lib, f).restype = ctypes.c_int
    _lib = lib
    return lib


def declared_functions() -> list:
    """Names of every entry point declared in the headers under include/."""
    names = set()
    for h in HEADERS:
        with open(h) as f:
            names |= set(re.findall(r"\b(commitkv_[a-z_]+)\s*\(", f.read()))
    return sorted(names)


def status_string(status: int) -> str:
    return load_library().commitkv_status_string(int(status)).decode()


def _check(rc: int, where: str):
    if rc != COMMITKV_OK:
        raise CommitKVError(rc, where)


# ----------------------------------------------------------------------------
# marshalling helpers (torch tensors -> pointers)


def _torch():
    import torch
    return torch


def _stream(stream) -> Optional[int]:
    torch = _torch()
    if stream is None:
        return torch.cuda.current_stream().cuda_stream or None
    if isinstance(stream, int):
        return stream or None
    return stream.cuda_stream or None


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr() if x.numel() else None


def _ptr_array(xs, n) -> Optional[ctypes.Array]:
    if xs is None:
        return None
    arr = (ctypes.c_void_p * n)()
    for i, x in enumerate(xs):
        arr[i] = _ptr(x)
    return arr


def _require_cuda(*ts):
    for t in ts:
        if t is not None and not isinstance(t, int) and t.numel() and not t.is_cuda:
            raise ValueError("CommitKV tensors must live on the GPU (no CPU fallback)")


@dataclass
class TrajTensors:
    """One trajectory's device tensors.

    k, v: [M][H][S][d] views (any strides with contiguous d); pos [S] int32;
    q [M][Hq][W][d] contiguous; q_pos [W] int32; page_start/page_len [P]."""
    k: object
    v: object
    pos: object
    q: object = None
    q_pos: object = None
    page_start: object = None
    page_len: object = None

    def desc(self) -> Traj:
        torch = _torch()
        k, v = self.k, self.v
        _require_cuda(k, v, self.pos, self.q, self.q_pos, self.page_start, self.page_len)
        assert k.dim() == 4 and k.stride() == v.stride() and k.shape == v.shape
        assert k.stride(3) == 1, "head_dim must be contiguous"
        for t in (self.pos, self.q_pos, self.page_start, self.page_len):
            assert t is None or t.dtype == torch.int32
        S = k.shape[2]
        W = 0 if self.q is None else self.q.shape[2]
        if self.q is not None:
            assert self.q.is_contiguous() and self.q.dtype == k.dtype
        P = 0 if self.page_start is None else self.page_start.numel()
        return Traj(_ptr(k), _ptr(v), k.stride(0), k.stride(1), k.stride(2), _ptr(self.pos), S,
                    _ptr(self.q), _ptr(self.q_pos), W, _ptr(self.page_start), _ptr(self.page_len), P)


def make_shape(M, H, Hq, d, dtype, softmax_scale=0.0) -> Shape:
    torch = _torch()
    code = {torch.float32: COMMITKV_F32, torch.bfloat16: COMMITKV_BF16}[dtype] \
        if not isinstance(dtype, int) else dtype
    return Shape(M, H, Hq, d, code, softmax_scale)


def _descs(trajs: Sequence[TrajTensors]):
    n = len(trajs)
    if not 1 <= n <= MAX_TRAJ:
        raise ValueError("1 <= n_traj <= 64")
    arr = (Traj * n)()
    for i, t in enumerate(trajs):
        arr[i] = t.desc()
    return arr


def _mask(layer_mask, M):
    if layer_mask is None:
        return None, None
    buf = (ctypes.c_uint8 * M)(*[1 if x else 0 for x in layer_mask])
    return buf, ctypes.cast(buf, ctypes.c_void_p)


# ----------------------------------------------------------------------------
# entry points


def commitkv_workspace_size(shape: Shape, trajs: Sequence[TrajTensors]) -> int:
    d = _descs(trajs)
    n = load_library().commitkv_workspace_size(ctypes.byref(shape), len(trajs), d)
    if n == 0:
        raise CommitKVError(COMMITKV_ERR_INVALID_ARG, "commitkv_workspace_size")
    return int(n)


def alloc_workspace(shape: Shape, trajs: Sequence[TrajTensors], device=None):
    """Allocate (with torch) and initialise a workspace for these trajectories."""
    torch = _torch()
    n = commitkv_workspace_size(shape, trajs)
    ws = torch.empty(n + 256, dtype=torch.uint8, device=device or "cuda")
    off = (-ws.data_ptr()) % 256
    ws = ws[off: off + n]
    commitkv_workspace_init(ws)
    return ws


def commitkv_workspace_init(ws, stream=None):
    _check(load_library().commitkv_workspace_init(_ptr(ws), ws.numel(), _stream(stream)),
           "commitkv_workspace_init")


def commitkv_workspace_status(ws, stream=None, clear: bool = True) -> int:
    return int(load_library().commitkv_workspace_status(_ptr(ws), ws.numel(), _stream(stream),
                                                        1 if clear else 0))


def commitkv_test_barrier_timeout(ws, blocks=2, stream=None):
    _check(load_library().commitkv_test_barrier_timeout(_ptr(ws), ws.numel(), int(blocks),
                                                        _stream(stream)),
           "commitkv_test_barrier_timeout")


def commitkv_page_effects(shape: Shape, trajs, R_out, head_R_out=None, stats_out=None,
                          layer_mask=None, workspace=None, stream=None):
    n = len(trajs)
    d = _descs(trajs)
    _mbuf, mptr = _mask(layer_mask, shape.layers)
    _require_cuda(*R_out)
    rc = load_library().commitkv_page_effects(
        ctypes.byref(shape), n, d, mptr, _ptr_array(R_out, n), _ptr_array(head_R_out, n),
        _ptr_array(stats_out, n), _ptr(workspace), workspace.numel(), _stream(stream))
    _check(rc, "commitkv_page_effects")


def commitkv_page_effects_from_stats(shape: Shape, trajs, stats_in, R_out, head_R_out=None,
                                     layer_mask=None, workspace=None, stream=None):
    n = len(trajs)
    d = _descs(trajs)
    _mbuf, mptr = _mask(layer_mask, shape.layers)
    _require_cuda(*R_out)
    rc = load_library().commitkv_page_effects_from_stats(
        ctypes.byref(shape), n, d, mptr, _ptr_array(stats_in, n), _ptr_array(R_out, n),
        _ptr_array(head_R_out, n), _ptr(workspace), workspace.numel(), _stream(stream))
    _check(rc, "commitkv_page_effects_from_stats")


def commitkv_token_scores(shape: Shape, trajs, stats, scores_out, layer_mask=None, workspace=None, stream=None):
    """Per-token fill scores (window attention with the given row stats)."""
    n = len(trajs)
    d = _descs(trajs)
    _mbuf, mptr = _mask(layer_mask, shape.layers)
    _require_cuda(*scores_out)
    rc = load_library().commitkv_token_scores(
        ctypes.byref(shape), n, d, mptr, _ptr_array(stats, n), _ptr_array(scores_out, n), _ptr(workspace),
        workspace.numel(), _stream(stream))
    _check(rc, "commitkv_token_scores")


def commitkv_classify(P, R_pre, R_post, eligible, state_out, cand_out, n_cand_out, workspace,
                      thresholds: Optional[Thresholds] = None, stream=None):
    n = len(P)
    Parr = (ctypes.c_int32 * n)(*[int(p) for p in P])
    rc = load_library().commitkv_classify(
        n, ctypes.cast(Parr, ctypes.c_void_p), _ptr_array(R_pre, n), _ptr_array(R_post, n),
        _ptr_array(eligible, n), ctypes.byref(thresholds) if thresholds else None,
        _ptr_array(state_out, n), _ptr_array(cand_out, n), _ptr(n_cand_out), _ptr(workspace),
        workspace.numel(), _stream(stream))
    _check(rc, "commitkv_classify")


COMMITKV_CLASSIFY_NO_PRECOMMIT = 1
COMMITKV_CLASSIFY_NO_PERCENTILE = 2


def commitkv_classify_variant(P, R_pre, R_post, eligible, variant, state_out, cand_out, n_cand_out,
                              workspace, thresholds: Optional[Thresholds] = None, stream=None):
    n = len(P)
    Parr = (ctypes.c_int32 * n)(*[int(p) for p in P])
    rc = load_library().commitkv_classify_variant(
        n, ctypes.cast(Parr, ctypes.c_void_p), _ptr_array(R_pre, n), _ptr_array(R_post, n),
        _ptr_array(eligible, n), ctypes.byref(thresholds) if thresholds else None, int(variant),
        _ptr_array(state_out, n), _ptr_array(cand_out, n), _ptr(n_cand_out), _ptr(workspace),
        workspace.numel(), _stream(stream))
    _check(rc, "commitkv_classify_variant")


def commitkv_joint_test(shape: Shape, post, stats, cand, n_cand, tau_joint, accepted_out,
                        step_R_out=None, layer_mask=None, workspace=None, stream=None):
    n = len(post)
    d = _descs(post)
    _mbuf, mptr = _mask(layer_mask, shape.layers)
    rc = load_library().commitkv_joint_test(
        ctypes.byref(shape), n, d, mptr, _ptr_array(stats, n), _ptr_array(cand, n), _ptr(n_cand),
        float(tau_joint), _ptr_array(accepted_out, n), _ptr_array(step_R_out, n), _ptr(workspace),
        workspace.numel(), _stream(stream))
    _check(rc, "commitkv_joint_test")


def commitkv_compact(shape: Shape, cache, retired, pending, pending_priority, fill_score, budget_B,
                     pending_tokens_BN, pending_cap_pages, idx_out, n_idx_out, k_out=None,
                     v_out=None, pos_out=None, workspace=None, stream=None):
    n = len(cache)
    d = _descs(cache)
    npend = (ctypes.c_int32 * n)(*[0 if p is None else int(p.numel()) for p in pending])
    rc = load_library().commitkv_compact(
        ctypes.byref(shape), n, d, _ptr_array(retired, n), _ptr_array(pending, n),
        ctypes.cast(npend, ctypes.c_void_p), _ptr_array(pending_priority, n),
        _ptr_array(fill_score, n), int(budget_B), int(pending_tokens_BN), int(pending_cap_pages),
        _ptr_array(idx_out, n), _ptr(n_idx_out), _ptr_array(k_out, n), _ptr_array(v_out, n),
        _ptr_array(pos_out, n), _ptr(workspace), workspace.numel(), _stream(stream))
    _check(rc, "commitkv_compact")


def commitkv_compact_in_place(shape: Shape, cache, retired, pending, pending_priority, fill_score, budget_B,
                              pending_tokens_BN, pending_cap_pages, idx_out, n_idx_out, workspace=None,
                              stream=None):
    """commitkv_compact with the gather inside the caches: K and V row I_j
    of every (layer, KV head) slice moves to row j of the same slice, and
    pos[j] = pos[I_j], for j < n_idx_out[t]; the caches' k, v and pos
    tensors are overwritten."""
    n = len(cache)
    d = _descs(cache)
    npend = (ctypes.c_int32 * n)(*[0 if p is None else int(p.numel()) for p in pending])
    rc = load_library().commitkv_compact_in_place(
        ctypes.byref(shape), n, d, _ptr_array(retired, n), _ptr_array(pending, n),
        ctypes.cast(npend, ctypes.c_void_p), _ptr_array(pending_priority, n),
        _ptr_array(fill_score, n), int(budget_B), int(pending_tokens_BN), int(pending_cap_pages),
        _ptr_array(idx_out, n), _ptr(n_idx_out), _ptr(workspace), workspace.numel(), _stream(stream))
    _check(rc, "commitkv_compact_in_place")


def commitkv_compact_noalloc(shape: Shape, cache, retired, pending, pending_priority, fill_score,
                             budget_B, pending_tokens_BN, pending_cap_pages, idx_out, n_idx_out,
                             k_out=None, v_out=None, pos_out=None, status_out=None, stream=None):
    """commitkv_compact with the library's fixed device scratch instead of a
    workspace, for callers that cannot allocate device memory when they
    compact.  Calls on one device share that scratch, so calls that can
    overlap on the GPU must be serialised; status_out (device int32 [1])
    receives the call's device-side status."""
    n = len(cache)
    d = _descs(cache)
    npend = (ctypes.c_int32 * n)(*[0 if p is None else int(p.numel()) for p in pending])
    rc = load_library().commitkv_compact_noalloc(
        ctypes.byref(shape), n, d, _ptr_array(retired, n), _ptr_array(pending, n),
        ctypes.cast(npend, ctypes.c_void_p), _ptr_array(pending_priority, n),
        _ptr_array(fill_score, n), int(budget_B), int(pending_tokens_BN), int(pending_cap_pages),
        _ptr_array(idx_out, n), _ptr(n_idx_out), _ptr_array(k_out, n), _ptr_array(v_out, n),
        _ptr_array(pos_out, n), _ptr(status_out), _stream(stream))
    _check(rc, "commitkv_compact_noalloc")
