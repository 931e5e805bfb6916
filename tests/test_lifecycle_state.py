"""Checkpoint / resume of the lifecycle session (CPU): the state between
commits round-trips through torch.save, and a resumed session continues
exactly as the original (appends cut the same pages with the same ids)."""
import io

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2608_07855_gb300 import commitkv as ck  # noqa: E402
from paper_2608_07855_gb300.lifecycle import Session  # noqa: E402


def _session():
    shape = ck.Shape(2, 2, 4, 64, ck.COMMITKV_BF16, 0.0)
    th = ck.Thresholds(1.0, 0.45, 0.75, 0.5)
    return Session(shape, 16, 96, 0.125, capacity=256, protect_cap=2, thresholds=th, tau_joint=0.3,
                   device="cpu")


def _tokens(rng, a, b):
    K = torch.from_numpy(rng.standard_normal((2, 2, b - a, 64)).astype(np.float32)).to(torch.bfloat16)
    V = torch.from_numpy(rng.standard_normal((2, 2, b - a, 64)).astype(np.float32)).to(torch.bfloat16)
    return K, V, torch.arange(a, b, dtype=torch.int32)


def _same(x, y):
    assert x.S == y.S and x.pages == y.pages and x.next_id == y.next_id
    assert x.R_pre == y.R_pre and x.measured == y.measured and x.retired == y.retired
    S = x.S
    assert torch.equal(x.K[:, :, :S], y.K[:, :, :S]) and torch.equal(x.V[:, :, :S], y.V[:, :, :S])
    assert torch.equal(x.pos[:S], y.pos[:S])


def test_state_round_trip_and_resume():
    rng = np.random.default_rng(0)
    a = _session()
    K, V, pos = _tokens(rng, 0, 100)
    a.append(K, V, pos, [("reason", 0, 20), ("call", 20, 30), ("obs", 50, 50)])
    # the host state a commit leaves behind
    ids = a.page_ids()
    a.R_pre = {pid: 0.1 * k for k, pid in enumerate(ids)}
    a.measured = ids[2:]
    a.retired = {ids[0]}
    buf = io.BytesIO()
    torch.save(a.state_dict(), buf)
    buf.seek(0)
    b = _session()
    b.load_state_dict(torch.load(buf))
    _same(a, b)
    # both continue alike
    K, V, pos = _tokens(rng, 100, 160)
    for s in (a, b):
        s.append(K, V, pos, [("call", 100, 25), ("obs", 125, 35)])
    _same(a, b)


def test_resume_refuses_other_settings_and_small_capacity():
    rng = np.random.default_rng(1)
    a = _session()
    K, V, pos = _tokens(rng, 0, 200)
    a.append(K, V, pos, [("obs", 0, 200)])
    st = a.state_dict()
    other = Session(a.shape, 32, 96, 0.125, capacity=256, protect_cap=2, thresholds=a.thresholds, tau_joint=0.3,
                    device="cpu")
    with pytest.raises(ValueError):
        other.load_state_dict(st)
    small = Session(a.shape, 16, 96, 0.125, capacity=128, protect_cap=2, thresholds=a.thresholds, tau_joint=0.3,
                    device="cpu")
    with pytest.raises(ValueError):
        small.load_state_dict(st)


def test_checkpoint_cadence_counter():
    """The decode cadence: append() counts decoded tokens, checkpoint_due()
    asks for a checkpoint once checkpoint_every of them are in and the
    cache is over budget, and the counter travels in state_dict (CPU: the
    device is the CPU, no library call is made)."""
    import torch
    from paper_2608_07855_gb300 import commitkv as ck
    from paper_2608_07855_gb300.lifecycle import Session
    shape = ck.Shape(1, 1, 1, 64, ck.COMMITKV_F32, 0.0)
    s = Session(shape, G=16, B=40, eta=0.125, capacity=200, checkpoint_every=32, device="cpu")
    z = torch.zeros(1, 1, 30, 64)
    s.append(z, z, torch.arange(30, dtype=torch.int32), [], decoded=30)
    assert not s.checkpoint_due()  # 30 < 32 decoded
    s.append(z, z, torch.arange(30, 60, dtype=torch.int32), [], decoded=2)
    assert s.checkpoint_due()  # 32 decoded, 60 > 40 resident
    st = s.state_dict()
    t = Session(shape, G=16, B=40, eta=0.125, capacity=200, checkpoint_every=32, device="cpu")
    t.load_state_dict(st)
    assert t.decoded_since == 32 and t.checkpoint_due()
    u = Session(shape, G=16, B=100, eta=0.125, capacity=200, checkpoint_every=32, device="cpu")
    u.append(z, z, torch.arange(30, dtype=torch.int32), [], decoded=40)
    assert not u.checkpoint_due()  # within budget
