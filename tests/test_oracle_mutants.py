"""The oracle's pins reject plausible mistakes (CPU only, no GPU).

Each case plants one mistake in a copy of the oracle -- a flipped sign, a
dropped term, an off-by-one causal mask, a query head read against the
wrong KV head, a swapped threshold, a reversed order -- and runs the pins of
test_oracle_pins.py against the copy: at least one of them must fail.  The
C part is rebuilt from a mutated copy of commitkv_oracle.c in a temporary
directory; the numpy part is re-executed from mutated source in a namespace
of its own.  The oracle itself is never changed.
"""
import inspect
import json
import os
import subprocess
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)

import test_oracle_pins as pins  # noqa: E402
from oracle import core  # noqa: E402

GOLDEN = os.path.join(HERE, "golden")


def _hand_cases():
    with open(os.path.join(GOLDEN, "effects_hand.json")) as f:
        return json.load(f)["cases"]


def _effect_pins():
    """The pins that constrain the C part: hand-derived values, sets and
    greedy scans, brute force over all subsets (an independent Python
    restatement), explicit deletion against the closed form, textbook and
    invariant cases."""
    cases = _hand_cases()
    return [
        ("hand effects, explicit", lambda: pins.test_hand_effects(cases, "explicit")),
        ("hand effects, closed form", lambda: pins.test_hand_effects(cases, "closed")),
        ("hand sets and greedy", lambda: pins.test_hand_sets_and_greedy(cases)),
        *[(f"brute force, seed {s}", (lambda s=s: pins.test_brute_force_all_subsets(s))) for s in range(4)],
        *[(f"explicit = closed, seed {s}", (lambda s=s: pins.test_explicit_equals_closed_form(s)))
          for s in range(3)],
        ("uniform attention", pins.test_uniform_attention_textbook),
        ("row stats textbook", pins.test_row_stats_textbook),
        ("invariants", pins.test_invariants),
    ]


def _selection_pins():
    return [
        ("token scores, uniform attention", pins.test_token_scores_uniform_attention),
        ("token scores, invariants", pins.test_token_scores_invariants),
        ("token scores, C row statistics", pins.test_token_scores_match_row_stats),
        ("classify hand table", lambda: pins.test_classify_hand(GOLDEN)),
        ("classify ablations hand table", lambda: pins.test_classify_variants_hand(GOLDEN)),
        *[(f"classify properties, seed {s}", (lambda s=s: pins.test_classify_properties(s))) for s in range(5)],
        ("selection hand table", lambda: pins.test_select_hand(GOLDEN)),
        *[(f"selection properties, seed {s}", (lambda s=s: pins.test_select_properties(s))) for s in range(6)],
    ]


def _failing(checks):
    failed = []
    for name, fn in checks:
        try:
            fn()
        except Exception:  # an assertion, or the mistake made the pin's own run fail
            failed.append(name)
    return failed


# (what the mistake is, the text it replaces in commitkv_oracle.c, the mistaken text)
C_MUTANTS = [
    ("the causal mask drops the query's own position",
     "vis[i] = pb->pos[i] <= pb->qpos[w];", "vis[i] = pb->pos[i] < pb->qpos[w];"),
    ("Eq. 6 adds the page's share instead of removing it",
     "o2[c] = (o[c] - o2[c]) / (1.0 - sa);", "o2[c] = (o[c] + o2[c]) / (1.0 - sa);"),
    ("Eq. 6 without the renormalisation by 1 - sum a",
     "o2[c] = (o[c] - o2[c]) / (1.0 - sa);", "o2[c] = o[c] - o2[c];"),
    ("the relative change is not divided by ||o||",
     "return sqrt(num) / sqrt(den);", "return sqrt(num);"),
    ("Eq. 7 sums over the window instead of taking the maximum",
     "if (r > Rh[E]) Rh[E] = r; /* Eq. 7: max over the window */", "Rh[E] += r;"),
    ("a query head reads the wrong KV head",
     "int g = pb->Hq / pb->H, kvh = h / g;\n  const double *q = q_row(pb, l, h, w);",
     "int g = pb->Hq / pb->H, kvh = h % pb->H;\n  const double *q = q_row(pb, l, h, w);"),
    ("the softmax scale is dropped",
     "s[i] = vis[i] ? pb->scale * dot(", "s[i] = vis[i] ? dot("),
    ("deleting every visible token gives 0 instead of rule (2)",
     "r = OKV_INF; /* rule (2) */", "r = 0.0; /* rule (2) */"),
    ("the greedy scan (explicit deletion) accepts only below tau",
     "    step_R[j] = R;\n    if (R <= tau) {\n      accepted[E] = 1;\n      memcpy(drop, trial, pb->S);",
     "    step_R[j] = R;\n    if (R < tau) {\n      accepted[E] = 1;\n      memcpy(drop, trial, pb->S);"),
    ("the greedy scan (closed form) accepts only below tau",
     "    step_R[j] = R;\n    if (R <= tau) {\n      accepted[E] = 1;\n      greedy_pass(&base, rows, nthreads, E, 1);",
     "    step_R[j] = R;\n    if (R < tau) {\n      accepted[E] = 1;\n      greedy_pass(&base, rows, nthreads, E, 1);"),
    ("the greedy scan (explicit deletion) forgets accepted pages",
     "      accepted[E] = 1;\n      memcpy(drop, trial, pb->S);", "      accepted[E] = 1;"),
    ("the greedy scan (closed form) does not fold accepted pages into D",
     "      accepted[E] = 1;\n      greedy_pass(&base, rows, nthreads, E, 1);", "      accepted[E] = 1;"),
]


@pytest.fixture(scope="module")
def c_source():
    with open(core._SRC) as f:
        return f.read()


@pytest.mark.parametrize("what,old,new", C_MUTANTS, ids=[m[0] for m in C_MUTANTS])
def test_pins_reject_c_mutant(what, old, new, c_source, tmp_path, monkeypatch):
    assert c_source.count(old) == 1, what
    src = tmp_path / "oracle_mutant.c"
    src.write_text(c_source.replace(old, new))
    so = tmp_path / "liboracle_mutant.so"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-o", str(so),
                           str(src), "-lm", "-lpthread"])
    monkeypatch.setattr(core, "_lib", None)
    monkeypatch.setattr(core, "build", lambda force=False: str(so))
    failed = _failing(_effect_pins())
    assert failed, f"no pin rejects the mistake: {what}"


def test_pins_accept_the_oracle(monkeypatch):
    """The same harness passes on the unmodified oracle (so a rejection
    above is the planted mistake's doing)."""
    assert _failing(_effect_pins()) == []
    assert _failing(_selection_pins()) == []


# (function, what the mistake is, the text it replaces, the mistaken text)
PY_MUTANTS = [
    ("classify", "the candidate state is the newly-active pattern (L- and H+)",
     "st[Hm & Lp] = STATE_CANDIDATE", "st[Lm & Hp] = STATE_CANDIDATE"),
    ("classify", "L+ tested against tau_use instead of tau_dead",
     "Lp = (Rp <= t_dead) & (Pp <= r_dead)", "Lp = (Rp <= t_use) & (Pp <= r_dead)"),
    ("classify", "H- without its percentile condition",
     "Hm = (Rm >= t_use) & (Pm >= r_use)", "Hm = (Rm >= t_use)"),
    ("classify", "candidates ordered by decreasing R+",
     "key=lambda E: (R_post[E], -R_pre[E], E)", "key=lambda E: (-R_post[E], -R_pre[E], E)"),
    ("percentile_ranks", "ties ranked at the upper end",
     "np.count_nonzero(Rc < x)", "np.count_nonzero(Rc <= x)"),
    ("protect_pending", "pending pages protected in increasing priority",
     "live.sort(key=lambda t: (-t[1], t[0]))", "live.sort(key=lambda t: (t[1], t[0]))"),
    ("protect_pending", "the page cap not applied",
     "if len(out) + 1 > cap_pages or tokens + int(page_len[E]) > B_N:",
     "if tokens + int(page_len[E]) > B_N:"),
    ("select_indices", "the fill keeps the lowest scores",
     "key=lambda i: (-float(fill_score[i]), -i)", "key=lambda i: (float(fill_score[i]), -i)"),
    ("select_indices", "retired pages not excluded",
     "tok_retired[page_start[E]: page_start[E] + page_len[E]] = True", "pass"),
    ("token_scores", "a token's weights summed over the rows instead of maximised",
     "score[idx] = np.maximum(score[idx], e / e.sum())", "score[idx] = score[idx] + e / e.sum()"),
    ("token_scores", "the weights not normalised by the row's sum",
     "score[idx] = np.maximum(score[idx], e / e.sum())", "score[idx] = np.maximum(score[idx], e)"),
    ("token_scores", "the causal mask drops the query's own position",
     "vis = pb.pos <= pb.qpos[w]", "vis = pb.pos < pb.qpos[w]"),
    ("token_scores", "a query head reads the wrong KV head",
     "Kh = pb.K[li, h // g]", "Kh = pb.K[li, h % pb.H]"),
]


@pytest.mark.parametrize("fn,what,old,new", PY_MUTANTS, ids=[f"{m[0]}: {m[1]}" for m in PY_MUTANTS])
def test_pins_reject_python_mutant(fn, what, old, new, monkeypatch):
    src = inspect.getsource(getattr(core, fn))
    assert src.count(old) == 1, what
    ns = dict(core.__dict__)
    exec(compile(src.replace(old, new), f"<mutant of {fn}>", "exec"), ns)
    monkeypatch.setattr(core, fn, ns[fn])
    failed = _failing(_selection_pins())
    assert failed, f"no pin rejects the mistake: {fn}: {what}"


# ----------------------------------------------------------------------------
# the multi-commit driver (Algorithm 1's outer loop)

import textwrap  # noqa: E402

import test_oracle_lifecycle as lpins  # noqa: E402
from oracle import lifecycle  # noqa: E402


def _lifecycle_pins():
    return [
        ("hand-worked timeline", lpins.test_hand_worked_timeline),
        ("hand-worked timeline, scan cap 0", lpins.test_hand_worked_timeline_scan_cap),
        ("timeline invariants", lpins.test_oracle_lifecycle_invariants),
        ("decode checkpoint after a commit", lpins.test_decode_checkpoint_after_a_commit_protects_nothing),
    ]


# (method of OracleSession, what the mistake is, the text it replaces, the mistaken text)
LIFECYCLE_MUTANTS = [
    ("post_commit", "every non-retired resident page is in E_c, the new observation's included",
     "eligible = np.asarray([pid in meas and pid not in self.retired for pid in ids], np.uint8)",
     "eligible = np.asarray([pid not in self.retired for pid in ids], np.uint8)"),
    ("post_commit", "the candidate list is not cut to the scan cap",
     "cand = cand[:self.scan_cap]", "cand = cand"),
    ("post_commit", "accepted pages do not join D_c",
     "self.retired |= set(accepted)", "pass"),
    ("pre_commit", "retired pages are measured again",
     "self.measured = [pid for pid in self.page_ids() if pid not in self.retired]",
     "self.measured = list(self.page_ids())"),
    ("checkpoint_resident", "a partly retained page keeps its old first row",
     "pages.append([pid, int(new_index[s + kept[0]]), len(kept)])",
     "pages.append([pid, int(new_index[s]), len(kept)])"),
    ("checkpoint_resident", "a partly retained page keeps its old length",
     "pages.append([pid, int(new_index[s + kept[0]]), len(kept)])",
     "pages.append([pid, int(new_index[s + kept[0]]), n])"),
    ("checkpoint_resident", "every non-retired page is protected as pending",
     "pend = [i for i, pid in enumerate(ids) if pid in set(self.measured)]",
     "pend = [i for i, pid in enumerate(ids) if pid not in self.retired]"),
]


@pytest.mark.parametrize("meth,what,old,new", LIFECYCLE_MUTANTS,
                         ids=[f"{m[0]}: {m[1]}" for m in LIFECYCLE_MUTANTS])
def test_pins_reject_lifecycle_mutant(meth, what, old, new, monkeypatch):
    src = textwrap.dedent(inspect.getsource(getattr(lifecycle.OracleSession, meth)))
    assert src.count(old) == 1, what
    ns = dict(lifecycle.__dict__)
    exec(compile(src.replace(old, new), f"<mutant of OracleSession.{meth}>", "exec"), ns)
    monkeypatch.setattr(lifecycle.OracleSession, meth, ns[meth])
    failed = _failing(_lifecycle_pins())
    assert failed, f"no pin rejects the mistake: {meth}: {what}"


def test_lifecycle_pins_accept_the_oracle():
    assert _failing(_lifecycle_pins()) == []
