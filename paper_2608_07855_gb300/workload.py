"""Device-resident synthetic trajectories and the CommitKV step.

A step is the whole hot path for every trajectory of a batch, as five
library calls on one stream:
  1. commitkv_page_effects  pre-commit cache,  Q-  -> R-         (Eq. 8)
  2. commitkv_page_effects  post-commit cache, Q+ -> R+, stats   (Eq. 8)
  3. commitkv_classify      R-, R+, E_c -> states, candidates     (Eq. 9-10)
  4. commitkv_joint_test    candidates  -> accepted (= D_c here)  (Eq. 11)
  5. commitkv_compact       D_c, pending (o_t's pages), fill      (Eq. 12-13, 4)
The pre-commit cache is a prefix view of the post-commit cache (the same
memory, as with cross-turn KV reuse).  Pending pages are the observation's
pages with their R+ standing in for the R- of the next commit (they have
no pre-commit measurement in a single step).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from . import commitkv as ck
from . import synth


def _torch():
    import torch
    return torch


@dataclass
class DeviceTrajectory:
    tr: synth.Trajectory
    K: object
    V: object
    pos: object
    Q_pre: object
    Q_post: object
    qpos_pre: object
    qpos_post: object
    page_start: object
    page_len: object
    eligible: object
    pending: object
    fill: object

    @classmethod
    def upload(cls, tr: synth.Trajectory, device="cuda"):
        torch = _torch()
        bf = tr.cfg.dtype == "bf16"

        def vals(a):
            t = torch.from_numpy(np.ascontiguousarray(a))
            if bf:
                t = t.view(torch.bfloat16)
            return t.to(device)

        def i32(a):
            return torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(device)

        return cls(tr, vals(tr.K), vals(tr.V), i32(tr.pos), vals(tr.Q_pre), vals(tr.Q_post),
                   i32(tr.qpos_pre), i32(tr.qpos_post), i32(tr.page_start), i32(tr.page_len),
                   torch.from_numpy(tr.eligible.astype(np.uint8)).to(device), i32(tr.pending),
                   torch.from_numpy(tr.fill_score).to(device))

    @property
    def P_pre(self):
        return self.tr.P_pre

    @property
    def P_post(self):
        return self.tr.P_post

    def pre(self) -> ck.TrajTensors:
        L = self.tr.L_pre
        return ck.TrajTensors(self.K[:, :, :L], self.V[:, :, :L], self.pos[:L], self.Q_pre,
                              self.qpos_pre, self.page_start[:self.P_pre], self.page_len[:self.P_pre])

    def post(self) -> ck.TrajTensors:
        return ck.TrajTensors(self.K, self.V, self.pos, self.Q_post, self.qpos_post,
                              self.page_start, self.page_len)


def shape_of(cfg: synth.Config) -> ck.Shape:
    return ck.Shape(cfg.M, cfg.H, cfg.Hq, cfg.d,
                    ck.COMMITKV_BF16 if cfg.dtype == "bf16" else ck.COMMITKV_F32, 0.0)


class StepBuffers:
    """Outputs of one step for a batch of device trajectories."""

    def __init__(self, cfg: synth.Config, trajs, device="cuda"):
        torch = _torch()
        self.cfg = cfg
        self.trajs = trajs
        self.shape = shape_of(cfg)
        f32, u8, i32 = torch.float32, torch.uint8, torch.int32
        self.R_pre = [torch.zeros(t.P_post, dtype=f32, device=device) for t in trajs]
        self.R_post = [torch.zeros(t.P_post, dtype=f32, device=device) for t in trajs]
        self.stats = [torch.zeros(cfg.M, cfg.Hq, cfg.W, cfg.d + 4, dtype=f32, device=device) for t in trajs]
        self.state = [torch.zeros(t.P_post, dtype=u8, device=device) for t in trajs]
        self.cand = [torch.zeros(max(t.P_post, 1), dtype=i32, device=device) for t in trajs]
        self.n_cand = torch.zeros(len(trajs), dtype=i32, device=device)
        self.accepted = [torch.zeros(max(t.P_post, 1), dtype=u8, device=device) for t in trajs]
        self.step_R = [torch.zeros(max(t.P_post, 1), dtype=f32, device=device) for t in trajs]
        self.idx = [torch.zeros(max(cfg.B, 1), dtype=i32, device=device) for t in trajs]
        self.n_idx = torch.zeros(len(trajs), dtype=i32, device=device)
        dt = trajs[0].K.dtype
        self.k_out = [torch.empty(cfg.M, cfg.H, cfg.B, cfg.d, dtype=dt, device=device) for t in trajs]
        self.v_out = [torch.empty(cfg.M, cfg.H, cfg.B, cfg.d, dtype=dt, device=device) for t in trajs]
        self.pos_out = [torch.empty(max(cfg.B, 1), dtype=i32, device=device) for t in trajs]
        # sized for the pre- and post-commit caches scored in one call
        self.ws = ck.alloc_workspace(self.shape, [t.pre() for t in trajs] + [t.post() for t in trajs],
                                     device=device)

    # the five calls ---------------------------------------------------------
    def score_pre(self, stream=None):
        ck.commitkv_page_effects(self.shape, [t.pre() for t in self.trajs],
                                 [r[:t.P_pre] for r, t in zip(self.R_pre, self.trajs)],
                                 workspace=self.ws, stream=stream)

    def score_post(self, stream=None):
        ck.commitkv_page_effects(self.shape, [t.post() for t in self.trajs], self.R_post,
                                 stats_out=self.stats, workspace=self.ws, stream=stream)

    def score(self, stream=None):
        """R- and R+ (and the post-commit stats) in one call: the pre- and
        post-commit caches of every trajectory form one batch, so the scoring
        kernels run once over both."""
        n = len(self.trajs)
        ck.commitkv_page_effects(self.shape, [t.pre() for t in self.trajs] + [t.post() for t in self.trajs],
                                 [r[:t.P_pre] for r, t in zip(self.R_pre, self.trajs)] + self.R_post,
                                 stats_out=[None] * n + self.stats, workspace=self.ws, stream=stream)

    def classify(self, stream=None):
        ck.commitkv_classify([t.P_post for t in self.trajs], self.R_pre, self.R_post,
                             [t.eligible for t in self.trajs], self.state, self.cand, self.n_cand,
                             self.ws, stream=stream)

    def joint(self, stream=None):
        ck.commitkv_joint_test(self.shape, [t.post() for t in self.trajs], self.stats, self.cand,
                               self.n_cand, self.cfg.tau_joint, self.accepted, self.step_R,
                               workspace=self.ws, stream=stream)

    def compact(self, stream=None):
        ck.commitkv_compact(self.shape, [t.post() for t in self.trajs], self.accepted,
                            [t.pending for t in self.trajs], self.R_post,
                            [t.fill for t in self.trajs], self.cfg.B, self.cfg.B_N,
                            self.cfg.pending_cap, self.idx, self.n_idx, self.k_out, self.v_out,
                            self.pos_out, workspace=self.ws, stream=stream)

    def step(self, stream=None):
        self.score(stream)
        self.classify(stream)
        self.joint(stream)
        self.compact(stream)

    def status(self, stream=None) -> int:
        return ck.commitkv_workspace_status(self.ws, stream)
