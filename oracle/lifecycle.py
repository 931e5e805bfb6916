"""Oracle of the multi-commit lifecycle (Algorithm 1's outer loop), fp64.

Test infrastructure: only tests/ may import this module.  It strings the
oracle's single-commit functions (oracle.core) together across tool-call
commits, in the order of Algorithm 1, with plain Python bookkeeping:

  pre_commit   commit c_t: the pages of every completed tool-call or
               observation event are measurable (E_{c_t}); R- over the
               pre-commit window (Eq. 5-8).  They wait for their post-commit
               measurement (pending, Section 3.3 "Protecting incomplete
               transitions").
  checkpoint   Eq. 12-13 and Eq. 4: the retired pages D_c are excluded, at
               most B_N = floor(eta B) tokens and at most cap pages of the
               pending ones are protected by decreasing R-, the budget B is
               filled by the caller's per-token score, and K, V, positions are
               gathered.  A page keeps the tokens of it that are retained; its
               span is found again from the retained indices.
  decode_checkpoint  the same on the decode cadence, the fill score being
               each resident token's largest attention weight from the latest
               window (reading 13b, core.token_scores).
  post_commit  R+ over the post-commit window; E_c = the pages measured at
               the pre-commit that are still resident and not retired;
               classification (Eq. 9-10), at most scan_cap candidates in
               order (the paper scans at most 64 pages per commit), the
               greedy joint test (Eq. 11); D_c gains the accepted pages.

Pages are identified by ids that survive compaction.  Events are cut into
pages as in Section 3.1: from the event's first token into G-token pages,
the last page taking the remainder; only tool-call and observation events
have pages.
"""
from __future__ import annotations

import math

import numpy as np

from oracle import core


class OracleSession:
    def __init__(self, M, H, Hq, d, G, B, eta, scan_cap=64, protect_cap=16, thresholds=None,
                 no_precommit=False, no_percentile=False, tau_joint=0.05):
        self.M, self.H, self.Hq, self.d, self.G = M, H, Hq, d, G
        self.B, self.B_N = B, int(math.floor(eta * B))
        self.scan_cap, self.protect_cap = scan_cap, protect_cap
        self.th = thresholds or dict(tau_use=0.05, tau_dead=0.01, rho_use=0.75, rho_dead=0.25)
        self.no_precommit, self.no_percentile, self.tau_joint = no_precommit, no_percentile, tau_joint
        self.K = np.zeros((M, H, 0, d))
        self.V = np.zeros((M, H, 0, d))
        self.pos = np.zeros(0, np.int64)
        self.pages = []          # [id, start, len] in resident order
        self.next_id = 0
        self.R_pre = {}          # page id -> R- of the latest commit
        self.measured = []       # page ids measured at the latest pre-commit, awaiting post
        self.retired = set()     # D_c: accepted page ids still resident
        self.log = []

    # ---------------------------------------------------------------- cache
    def append(self, K, V, pos, events):
        """Append resident tokens (K, V [M][H][n][d] float64, absolute
        positions [n]) and cut their tool-call / observation events into
        pages; events = [(kind, first token, length)] in timeline positions."""
        S0 = self.pos.shape[0]
        self.K = np.concatenate([self.K, K], axis=2)
        self.V = np.concatenate([self.V, V], axis=2)
        self.pos = np.concatenate([self.pos, np.asarray(pos, np.int64)])
        p0 = int(pos[0]) if len(pos) else 0
        for kind, b, n in events:
            if kind not in ("call", "obs"):
                continue
            for s in range(b, b + n, self.G):
                self.pages.append([self.next_id, S0 + (s - p0), min(self.G, b + n - s)])
                self.next_id += 1

    def _problem(self, Q, qpos):
        ps = np.asarray([p[1] for p in self.pages], np.int32)
        pl = np.asarray([p[2] for p in self.pages], np.int32)
        return core.Problem(self.K, self.V, self.pos.astype(np.int32), Q, np.asarray(qpos, np.int32), ps, pl)

    def page_ids(self):
        return [p[0] for p in self.pages]

    # ---------------------------------------------------------------- commit
    def pre_commit(self, Q, qpos):
        """R- of every resident page over the pre-commit window; the
        non-retired ones become E_{c_t} and wait for their post measurement."""
        pb = self._problem(Q, qpos)
        R, _ = core.page_effects(pb, "closed")
        self.R_pre = {pid: float(R[i]) for i, pid in enumerate(self.page_ids())}
        self.measured = [pid for pid in self.page_ids() if pid not in self.retired]
        self.log.append(("pre", R.copy()))
        return R

    # ---------------------------------------------------------------- checkpoint
    def checkpoint(self, fill_by_pos):
        """Eq. 12-13 and Eq. 4 at a compression checkpoint, the budget filled
        by a score per absolute position: returns I (old resident indices,
        ascending)."""
        return self.checkpoint_resident(np.asarray(fill_by_pos, np.float32)[self.pos])

    def fill_scores(self, Q, qpos):
        """The self-contained fill score of every resident token (reading
        13b): its largest attention weight from the window (Q, qpos)."""
        return core.token_scores(self._problem(Q, qpos))

    def decode_checkpoint(self, Q, qpos):
        """A checkpoint on the decode cadence (the paper compresses every 128
        decoded tokens), the budget filled by the window's attention."""
        return self.checkpoint_resident(self.fill_scores(Q, qpos))

    def checkpoint_resident(self, fill):
        """Eq. 12-13 and Eq. 4 with a fill score per resident token."""
        S = self.pos.shape[0]
        ids = self.page_ids()
        ps = np.asarray([p[1] for p in self.pages], np.int64)
        pl = np.asarray([p[2] for p in self.pages], np.int64)
        retired = np.asarray([pid in self.retired for pid in ids], np.uint8)
        pend = [i for i, pid in enumerate(ids) if pid in set(self.measured)]
        prio = np.asarray([self.R_pre[ids[i]] for i in pend], np.float32)
        fill = np.asarray(fill, np.float32)
        I = core.select_indices(S, ps, pl, retired, np.asarray(pend, np.int64), prio, fill, self.B, self.B_N,
                                self.protect_cap)
        self.K, self.V, pos = core.gather(self.K, self.V, self.pos, I)
        self.pos = np.asarray(pos, np.int64)
        keep = np.zeros(S, bool)
        keep[I] = True
        new_index = np.cumsum(keep) - 1
        pages = []
        for pid, s, n in self.pages:
            kept = np.flatnonzero(keep[s:s + n])
            if len(kept) == 0:
                continue  # gone, retired ones included
            pages.append([pid, int(new_index[s + kept[0]]), len(kept)])
        self.pages = pages
        alive = set(self.page_ids())
        self.retired &= alive
        self.log.append(("checkpoint", np.asarray(I)))
        return np.asarray(I)

    # ---------------------------------------------------------------- post
    def post_commit(self, Q, qpos):
        """Decisions of the latest commit: returns (R+ per resident page,
        candidates and accepted pages as page ids, the joint effects)."""
        pb = self._problem(Q, qpos)
        Rp, _ = core.page_effects(pb, "closed")
        ids = self.page_ids()
        meas = set(self.measured)
        eligible = np.asarray([pid in meas and pid not in self.retired for pid in ids], np.uint8)
        Rm = np.asarray([self.R_pre.get(pid, 0.0) if eligible[i] else 0.0 for i, pid in enumerate(ids)])
        # later stages take fp32 effects, as the library's interface does
        Rm32, Rp32 = Rm.astype(np.float32), Rp.astype(np.float32)
        state, cand = core.classify(Rm32, Rp32, eligible, **self.th, no_precommit=self.no_precommit,
                                    no_percentile=self.no_percentile)
        cand = cand[:self.scan_cap]
        acc, step = core.greedy(pb, cand, self.tau_joint, "closed", stats=core.row_stats(pb))
        accepted = [ids[E] for E in cand if acc[E]]
        self.retired |= set(accepted)
        self.measured = []
        out = dict(R_post=Rp, R_pre=Rm, cand=[ids[E] for E in cand], accepted=accepted, step_R=np.asarray(step),
                   eligible=[pid for i, pid in enumerate(ids) if eligible[i]], state=np.asarray(state))
        self.log.append(("post", out))
        return out
