"""Multi-commit lifecycle driver (Algorithm 1's outer loop) over the C ABI.

A Session holds one agent's resident KV cache on the device (K, V
[M][H][capacity][d], absolute positions) and the page table, and runs the
library's entry points in the order of Algorithm 1:

  append       new tokens (decoded reasoning and tool calls, prefilled
               observations); tool-call and observation events are cut into
               pages from their first token, G tokens per page, the last page
               taking the remainder (Section 3.1).
  pre_commit   commit c_t: R- of every resident page over the pre-commit
               window (commitkv_page_effects); the non-retired pages form
               E_{c_t} and wait for their post-commit measurement.
  checkpoint   commitkv_compact_in_place: the retired pages D_c are
               dropped, at most B_N = floor(eta B) tokens / protect_cap pages
               of the waiting pages are kept by decreasing R- (Eq. 12), the
               budget B is filled by the caller's per-token score (Eq. 13),
               and K, V and positions are gathered (Eq. 4) inside the
               session's own buffers; page spans are found again from the
               retained indices (a page keeps whichever of its tokens are
               retained, which stay contiguous).
  decode checkpoints  the paper's setting compresses every 128 decoded
               tokens: append() counts the decoded tokens, checkpoint_due()
               says when, and decode_checkpoint() fills the budget by each
               resident token's largest attention weight from the latest
               window (commitkv_token_scores on the window's row stats).
  post_commit  R+ over the post-commit window with the row stats;
               classification (Eq. 9-10, or an ablation variant of Section
               4.4); at most scan_cap candidates in order (the paper scans at
               most 64 pages per commit); the greedy joint test (Eq. 11);
               D_c gains the accepted pages.

state_dict / load_state_dict carry the state between commits (the resident
cache, the page table, R- of the latest pre-commit, the pages waiting for
their post-commit measurement, D_c) for checkpoint and resume.

Every computation runs in the library's kernels; this module keeps the page
table and the buffers.  The host reads back small per-commit results (page
effects, candidate counts, accepted masks, retained indices) to keep the page
table, once per call.
"""
from __future__ import annotations

import math

from . import commitkv as ck


def _torch():
    import torch
    return torch


class Session:
    def __init__(self, shape: ck.Shape, G: int, B: int, eta: float, capacity: int, scan_cap: int = 64,
                 protect_cap: int = 16, thresholds: ck.Thresholds = None, variant: int = 0,
                 tau_joint: float = 0.05, checkpoint_every: int = 128, device="cuda"):
        torch = _torch()
        self.shape, self.G, self.B = shape, G, B
        self.B_N = int(math.floor(eta * B))
        self.cap, self.scan_cap, self.protect_cap = capacity, scan_cap, protect_cap
        self.thresholds, self.variant, self.tau_joint = thresholds, variant, tau_joint
        self.dev = device
        dt = torch.bfloat16 if shape.dtype == ck.COMMITKV_BF16 else torch.float32
        M, H, d = shape.layers, shape.kv_heads, shape.head_dim
        self.K = torch.zeros(M, H, capacity, d, dtype=dt, device=device)
        self.V = torch.zeros(M, H, capacity, d, dtype=dt, device=device)
        self.pos = torch.zeros(capacity, dtype=torch.int32, device=device)
        self.S = 0
        self.pages = []       # [id, start, len] in resident order
        self.next_id = 0
        self.R_pre = {}       # page id -> R- (fp32) of the latest commit
        self.measured = []    # page ids waiting for their post-commit measurement
        self.retired = set()  # D_c: accepted page ids still resident
        self.checkpoint_every = checkpoint_every  # decoded tokens between checkpoints (0: caller-driven only)
        self.decoded_since = 0  # decoded tokens appended since the last checkpoint
        self.ws = None

    # ---------------------------------------------------------------- helpers
    def _traj(self, Q=None, qpos=None) -> ck.TrajTensors:
        torch = _torch()
        ps = torch.tensor([p[1] for p in self.pages], dtype=torch.int32, device=self.dev)
        pl = torch.tensor([p[2] for p in self.pages], dtype=torch.int32, device=self.dev)
        S = self.S
        return ck.TrajTensors(self.K[:, :, :S], self.V[:, :, :S], self.pos[:S], Q, qpos, ps, pl)

    def _workspace(self, traj):
        need = ck.commitkv_workspace_size(self.shape, [traj])
        if self.ws is None or self.ws.numel() < need:
            self.ws = ck.alloc_workspace(self.shape, [traj], device=self.dev)
        return self.ws

    def _check(self):
        st = ck.commitkv_workspace_status(self.ws)
        if st != ck.COMMITKV_OK:
            raise RuntimeError(f"device status: {ck.status_string(st)}")

    def page_ids(self):
        return [p[0] for p in self.pages]

    # ---------------------------------------------------------------- resume
    def state_dict(self):
        """Everything the session carries from one commit to the next: the
        resident cache (K, V, positions of its S tokens), the page table, R-
        of the latest pre-commit, the pages waiting for their post-commit
        measurement and D_c.  Tensors are copies on the session's device;
        torch.save writes the dict."""
        S = self.S
        return {
            "config": self._config(),
            "K": self.K[:, :, :S].clone(), "V": self.V[:, :, :S].clone(), "pos": self.pos[:S].clone(),
            "pages": [list(p) for p in self.pages], "next_id": self.next_id,
            "R_pre": dict(self.R_pre), "measured": list(self.measured), "retired": sorted(self.retired),
            "decoded_since": self.decoded_since,
        }

    def load_state_dict(self, st):
        """Resumes from state_dict() of a session with the same model shape,
        page size, budget and decision settings; the resident cache must fit
        this session's capacity."""
        if st["config"] != self._config():
            raise ValueError("state of a session with other settings")
        S = int(st["pos"].shape[0])
        if S > self.cap:
            raise ValueError("session capacity exceeded")
        self.K[:, :, :S].copy_(st["K"])
        self.V[:, :, :S].copy_(st["V"])
        self.pos[:S].copy_(st["pos"])
        self.S = S
        self.pages = [list(p) for p in st["pages"]]
        self.next_id = int(st["next_id"])
        self.R_pre = dict(st["R_pre"])
        self.measured = list(st["measured"])
        self.retired = set(st["retired"])
        self.decoded_since = int(st.get("decoded_since", 0))

    def _config(self):
        s, th = self.shape, self.thresholds
        return {"shape": (s.layers, s.kv_heads, s.q_heads, s.head_dim, s.dtype, float(s.softmax_scale)),
                "G": self.G, "B": self.B, "B_N": self.B_N, "scan_cap": self.scan_cap,
                "protect_cap": self.protect_cap, "variant": int(self.variant), "tau_joint": float(self.tau_joint),
                "checkpoint_every": int(self.checkpoint_every),
                "thresholds": None if th is None else (th.tau_use, th.tau_dead, th.rho_use, th.rho_dead)}

    # ---------------------------------------------------------------- cache
    def append(self, K, V, pos, events, decoded: int = 0):
        """Append n resident tokens: K, V [M][H][n][d] and absolute
        positions [n] (device tensors); events = [(kind, first position,
        length)] of the tool calls and observations inside them; decoded =
        how many of the n the model decoded (reasoning, tool calls), for the
        checkpoint cadence."""
        self.decoded_since += int(decoded)
        n = int(pos.shape[0])
        if self.S + n > self.cap:
            raise ValueError("session capacity exceeded")
        S0, p0 = self.S, int(pos[0]) if n else 0
        self.K[:, :, S0:S0 + n].copy_(K)
        self.V[:, :, S0:S0 + n].copy_(V)
        self.pos[S0:S0 + n].copy_(pos)
        self.S += n
        for kind, b, m in events:
            if kind not in ("call", "obs"):
                continue
            for s in range(b, b + m, self.G):
                self.pages.append([self.next_id, S0 + (s - p0), min(self.G, b + m - s)])
                self.next_id += 1

    # ---------------------------------------------------------------- commit
    def pre_commit(self, Q, qpos):
        """R- (device float [P]) of every resident page over the pre-commit
        window Q [M][Hq][W][d], qpos [W]; the non-retired pages wait for their
        post-commit measurement."""
        torch = _torch()
        tr = self._traj(Q, qpos)
        ws = self._workspace(tr)
        R = torch.zeros(max(len(self.pages), 1), device=self.dev)
        ck.commitkv_page_effects(self.shape, [tr], [R[:len(self.pages)]], workspace=ws)
        self._check()
        Rh = R[:len(self.pages)].cpu().tolist()
        ids = self.page_ids()
        self.R_pre = dict(zip(ids, Rh))
        self.measured = [pid for pid in ids if pid not in self.retired]
        return R[:len(self.pages)]

    def checkpoint_due(self) -> bool:
        """Whether the decode cadence calls for a checkpoint now: at least
        checkpoint_every decoded tokens since the last one (the paper's
        setting compresses every 128 decoded tokens) and more resident
        tokens than the budget."""
        return self.checkpoint_every > 0 and self.decoded_since >= self.checkpoint_every and self.S > self.B

    def fill_scores(self, Q, qpos):
        """Self-contained fill scores (device float [S]): each resident
        token's largest attention weight from the window Q [M][Hq][W][d],
        qpos [W] (commitkv_page_effects on the cache without pages for the
        window's row stats, then commitkv_token_scores)."""
        torch = _torch()
        s = self.shape
        S = self.S
        none = torch.zeros(0, dtype=torch.int32, device=self.dev)
        tr = ck.TrajTensors(self.K[:, :, :S], self.V[:, :, :S], self.pos[:S], Q, qpos, none, none)
        ws = self._workspace(self._traj())
        stats = torch.zeros(s.layers, s.q_heads, Q.shape[2], s.head_dim + 4, device=self.dev)
        R = torch.zeros(1, device=self.dev)
        ck.commitkv_page_effects(s, [tr], [R], stats_out=[stats], workspace=ws)
        scores = torch.zeros(max(S, 1), device=self.dev)
        ck.commitkv_token_scores(s, [tr], [stats], [scores[:S]], workspace=ws)
        self._check()
        return scores[:S]

    def decode_checkpoint(self, Q, qpos):
        """A checkpoint on the decode cadence, the budget filled by the
        window's attention (fill_scores).  Returns the retained indices."""
        return self.checkpoint(self.fill_scores(Q, qpos))

    def checkpoint(self, fill):
        """Compression checkpoint (Eq. 12-13, Eq. 4): fill = device float
        [S] per resident token.  Returns the retained resident indices I
        (device int32, ascending)."""
        torch = _torch()
        tr = self._traj()
        ws = self._workspace(tr)
        ids = self.page_ids()
        P, B = len(ids), self.B
        retired = torch.tensor([1 if pid in self.retired else 0 for pid in ids], dtype=torch.uint8,
                               device=self.dev)
        wait = set(self.measured)
        pend = [i for i, pid in enumerate(ids) if pid in wait]
        pending = torch.tensor(pend, dtype=torch.int32, device=self.dev)
        prio_p = torch.zeros(max(P, 1), dtype=torch.float32, device=self.dev)
        if P:
            prio_p[:P] = torch.tensor([self.R_pre.get(pid, 0.0) for pid in ids], dtype=torch.float32)
        idx = torch.full((max(B, 1),), -1, dtype=torch.int32, device=self.dev)
        n_idx = torch.zeros(1, dtype=torch.int32, device=self.dev)
        ck.commitkv_compact_in_place(self.shape, [tr], [retired], [pending], [prio_p], [fill[:self.S]], B,
                                     self.B_N, self.protect_cap, [idx], n_idx, workspace=ws)
        self._check()
        n = int(n_idx[0])
        I = idx[:n].cpu().tolist()
        # page spans from the retained indices
        new_index = {old: new for new, old in enumerate(I)}
        pages = []
        for pid, s, m in self.pages:
            kept = [new_index[i] for i in range(s, s + m) if i in new_index]
            if kept:
                pages.append([pid, kept[0], len(kept)])
        self.pages, self.S = pages, n
        self.retired &= set(self.page_ids())
        self.decoded_since = 0
        return idx[:n]

    def post_commit(self, Q, qpos):
        """Decisions of the latest commit over the post-commit window:
        returns dict(R_post (device [P]), cand, accepted (page ids in scan
        order / accepted ones), step_R (host list, one per scanned
        candidate))."""
        torch = _torch()
        tr = self._traj(Q, qpos)
        ws = self._workspace(tr)
        ids = self.page_ids()
        P = len(ids)
        s = self.shape
        Rp = torch.zeros(max(P, 1), device=self.dev)
        stats = torch.zeros(s.layers, s.q_heads, Q.shape[2], s.head_dim + 4, device=self.dev)
        ck.commitkv_page_effects(s, [tr], [Rp[:P]], stats_out=[stats], workspace=ws)
        wait = set(self.measured)
        el = [1 if (pid in wait and pid not in self.retired) else 0 for pid in ids]
        eligible = torch.tensor(el + [0] * (P == 0), dtype=torch.uint8, device=self.dev)
        Rm = torch.tensor([self.R_pre.get(pid, 0.0) if el[i] else 0.0 for i, pid in enumerate(ids)] + [0.0] * (P == 0),
                          dtype=torch.float32, device=self.dev)
        state = torch.zeros(max(P, 1), dtype=torch.uint8, device=self.dev)
        cand = torch.zeros(max(P, 1), dtype=torch.int32, device=self.dev)
        n_cand = torch.zeros(1, dtype=torch.int32, device=self.dev)
        ck.commitkv_classify_variant([P], [Rm], [Rp], [eligible], self.variant, [state], [cand], n_cand, ws,
                                     thresholds=self.thresholds)
        self._check()
        nc = min(int(n_cand[0]), self.scan_cap)  # the scan cap of the paper's setting
        n_scan = torch.tensor([nc], dtype=torch.int32, device=self.dev)
        acc = torch.zeros(max(P, 1), dtype=torch.uint8, device=self.dev)
        step = torch.zeros(max(P, 1), dtype=torch.float32, device=self.dev)
        ck.commitkv_joint_test(s, [tr], [stats], [cand], n_scan, self.tau_joint, [acc], [step], workspace=ws)
        self._check()
        c = cand[:nc].cpu().tolist()
        a = acc[:P].cpu().tolist()
        accepted = [ids[E] for E in c if a[E]]
        self.retired |= set(accepted)
        self.measured = []
        return dict(R_post=Rp[:P], cand=[ids[E] for E in c], accepted=accepted, step_R=step[:nc].cpu().tolist())
