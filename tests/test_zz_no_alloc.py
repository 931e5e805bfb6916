"""commitkv_compact_noalloc against commitkv_compact.

commitkv_compact_noalloc is for callers that cannot allocate device memory
when they compact: a serving engine that has reserved nearly all device
memory for its own KV pool (a later cudaMalloc fails, or must go through an
allocator a plug-in cannot reach), or a decode loop that cannot afford the
device-wide synchronisation of cudaFree.  Instead of a workspace it uses a
fixed scratch array that the library keeps on the GPU, shared by every call
and keeping the previous call's contents.  The GPU tests here make two calls
in a row (the second one finds the first one's leftovers in the scratch) and
require results bit-exact with the workspace entry point on the same inputs,
the tolerance every selection and gather test uses.

The file name makes pytest collect it last, so a failure here comes after
every other test has run.
"""
import ctypes

import pytest

from paper_2608_07855_gb300 import commitkv as ck

SCRATCH_BYTES = 4 << 20


def _header_limit():
    import re
    with open(ck.HEADERS[0]) as f:
        m = re.search(r"#define COMMITKV_NOALLOC_SCRATCH_BYTES \((\d+)u << (\d+)\)", f.read())
    return int(m.group(1)) << int(m.group(2))


def _fake_traj(S):
    """A descriptor with non-null but never dereferenced pointers: the size
    check refuses it on the host, before any CUDA call."""
    t = ck.Traj()
    t.k = t.v = t.pos = 256
    t.stride_layer, t.stride_head, t.stride_tok = 64 * S, 64 * S, 64
    t.S, t.W, t.P = S, 0, 0
    return t


def _call_raw(trajs, B=16, shape=None, workspace_entry=False):
    """commitkv_compact_noalloc (or, with workspace_entry, commitkv_compact
    with a fake workspace) on descriptors that only the host checks read."""
    lib = ck.load_library()
    n = len(trajs)
    arr = (ck.Traj * n)(*trajs)
    shape = shape or ck.make_shape(1, 1, 1, 64, ck.COMMITKV_F32)
    ptrs = (ctypes.c_void_p * n)(*([256] * n))
    npend = (ctypes.c_int32 * n)()
    if workspace_entry:
        return lib.commitkv_compact(ctypes.byref(shape), n, arr, ptrs, None,
                                    ctypes.cast(npend, ctypes.c_void_p), None, ptrs, B, 0, 0,
                                    ptrs, 256, None, None, None, 256, 1 << 20, None)
    return lib.commitkv_compact_noalloc(ctypes.byref(shape), n, arr, ptrs, None,
                                        ctypes.cast(npend, ctypes.c_void_p), None, ptrs, B, 0, 0,
                                        ptrs, 256, None, None, None, None, None)


def test_scratch_limit_matches_header():
    assert _header_limit() == SCRATCH_BYTES


def test_sizes_beyond_scratch_are_refused():
    """256 + sum of S_t rounded up to 256 must fit the 4 MiB array."""
    assert _call_raw([_fake_traj(SCRATCH_BYTES - 256 + 1)]) == ck.COMMITKV_ERR_WORKSPACE
    assert _call_raw([_fake_traj(SCRATCH_BYTES // 2)] * 2) == ck.COMMITKV_ERR_WORKSPACE
    assert _call_raw([_fake_traj(SCRATCH_BYTES)] * 3) == ck.COMMITKV_ERR_WORKSPACE


def test_host_checks_match_workspace_entry_point():
    """Both compaction entry points share one set of host-side checks: shapes
    and descriptors that commitkv_compact refuses, the no-alloc call refuses
    with the same code, before any CUDA call."""
    over_heads = ck.make_shape(2, 1, (1 << 19) + 1, 64, ck.COMMITKV_F32)  # layers * q_heads > 2^20
    bad_dim = ck.make_shape(1, 1, 1, 96, ck.COMMITKV_F32)
    bad_gqa = ck.make_shape(1, 2, 3, 64, ck.COMMITKV_F32)
    small = _fake_traj(1024)
    short = _fake_traj(1024)
    short.stride_tok = 32  # below head_dim
    cases = [(over_heads, [small], 16), (bad_dim, [small], 16), (bad_gqa, [small], 16),
             (None, [short], 16), (None, [small], -1)]
    for shape, trajs, B in cases:
        want = _call_raw(trajs, B, shape, workspace_entry=True)
        assert want in (ck.COMMITKV_ERR_INVALID_ARG, ck.COMMITKV_ERR_UNSUPPORTED)
        assert _call_raw(trajs, B, shape) == want


# ---------------------------------------------------------------------------
# GPU: two calls in a row against the workspace entry point


def _gpu():
    torch = pytest.importorskip("torch")
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    ck.load_library()
    return torch


def _batch(cfgs_seeds):
    from paper_2608_07855_gb300 import synth
    from paper_2608_07855_gb300.workload import DeviceTrajectory
    devs = [DeviceTrajectory.upload(synth.make_trajectory(c, s)) for c, s in cfgs_seeds]
    return cfgs_seeds[0][0], devs


class Call:
    """Inputs and two sets of outputs (workspace / no-alloc) of one compaction."""

    def __init__(self, torch, cfg, devs, seed, B, nan_fill=False):
        from paper_2608_07855_gb300.workload import shape_of
        g = torch.Generator().manual_seed(seed)
        self.shape = shape_of(cfg)
        self.cache = [d.post() for d in devs]
        self.retired = [(torch.rand(d.P_post, generator=g) < 0.25).to(torch.uint8).cuda()
                        for d in devs]
        self.pending = [d.pending for d in devs]
        self.prio = [torch.rand(d.P_post, generator=g).cuda() for d in devs]
        self.fill = [d.fill.clone() for d in devs]
        if nan_fill:
            self.fill[0][3] = float("nan")
        self.B, self.B_N, self.cap = B, int(cfg.eta * B), cfg.pending_cap
        self.out = [self._outputs(torch, cfg, devs) for _ in range(2)]

    def _outputs(self, torch, cfg, devs):
        n = len(devs)
        dt = devs[0].K.dtype
        return dict(
            idx=[torch.full((max(self.B, 1),), -1, dtype=torch.int32, device="cuda") for _ in devs],
            n_idx=torch.full((n,), -1, dtype=torch.int32, device="cuda"),
            k=[torch.zeros(cfg.M, cfg.H, self.B, cfg.d, dtype=dt, device="cuda") for _ in devs],
            v=[torch.zeros(cfg.M, cfg.H, self.B, cfg.d, dtype=dt, device="cuda") for _ in devs],
            pos=[torch.full((max(self.B, 1),), -1, dtype=torch.int32, device="cuda") for _ in devs],
            status=torch.full((1,), -1, dtype=torch.int32, device="cuda"))

    def args(self, o):
        return (self.shape, self.cache, self.retired, self.pending, self.prio, self.fill, self.B,
                self.B_N, self.cap, o["idx"], o["n_idx"], o["k"], o["v"], o["pos"])

    def run_noalloc(self):
        o = self.out[1]
        ck.commitkv_compact_noalloc(*self.args(o), status_out=o["status"])

    def run_workspace(self, torch):
        o = self.out[0]
        ws = ck.alloc_workspace(self.shape, self.cache)
        ck.commitkv_compact(*self.args(o), workspace=ws)
        o["status"].fill_(ck.commitkv_workspace_status(ws))

    def check(self, torch, want_status=ck.COMMITKV_OK):
        torch.cuda.synchronize()
        a, b = self.out
        assert int(a["status"][0]) == want_status
        assert int(b["status"][0]) == want_status
        if want_status != ck.COMMITKV_OK:
            return
        assert torch.equal(a["n_idx"], b["n_idx"])
        for t in range(len(self.cache)):
            n = int(a["n_idx"][t])
            assert 0 < n <= self.B
            assert torch.equal(a["idx"][t][:n], b["idx"][t][:n])
            assert torch.equal(a["pos"][t][:n], b["pos"][t][:n])
            # compare raw bits (torch.equal on floats would treat NaN != NaN)
            for key in ("k", "v"):
                x, y = a[key][t][:, :, :n], b[key][t][:, :, :n]
                iv = torch.int16 if x.dtype == torch.bfloat16 else torch.int32
                assert torch.equal(x.contiguous().view(iv), y.contiguous().view(iv))


@pytest.mark.gpu
def test_two_calls_in_a_row_match_workspace_entry_point():
    """A bf16 batch of two trajectories of different lengths, then an fp32
    trajectory with another head width and budget: the second call runs on
    the scratch the first one left behind."""
    torch = _gpu()
    from paper_2608_07855_gb300 import synth
    cfg1, devs1 = _batch([(synth.small_config(), 0),
                          (synth.small_config("small_long_pages", G=100, L_pre=900, L_obs=80,
                                              B=400), 4)])
    cfg2, devs2 = _batch([(synth.CONFIGS["tiny"], 1)])
    first = Call(torch, cfg1, devs1, seed=11, B=300)
    second = Call(torch, cfg2, devs2, seed=12, B=700)
    first.run_noalloc()
    second.run_noalloc()
    first.run_workspace(torch)
    second.run_workspace(torch)
    first.check(torch)
    second.check(torch)


@pytest.mark.gpu
def test_status_word_is_cleared_between_calls():
    """A NaN fill score is a device-side input error; the next call on the
    same scratch starts from a clean status word and matches again."""
    torch = _gpu()
    from paper_2608_07855_gb300 import synth
    cfg, devs = _batch([(synth.small_config(), 2)])
    bad = Call(torch, cfg, devs, seed=21, B=256, nan_fill=True)
    good = Call(torch, cfg, devs, seed=22, B=256)
    bad.run_noalloc()
    good.run_noalloc()
    bad.run_workspace(torch)
    good.run_workspace(torch)
    bad.check(torch, want_status=ck.COMMITKV_ERR_DEVICE_INPUT)
    good.check(torch)
