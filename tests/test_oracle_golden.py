"""The oracle's decoding loop (Algorithm 1, Sec. 3.2; Eq. 3-4) against hand-derived traces (no GPU).

The transformer is replaced by a scripted toy predictor (tests/toy_decode.py) and the
draft injection by a scripted corruption list, so that every iteration's rows, accepted counts,
pseudo-accepted counts, winner and committed tokens can be worked out by hand. The traces under
tests/golden/ were derived that way from the rules; this test runs the oracle's loop on the same
scripts and compares iteration by iteration. The toy cache checks that the committed rows extend the
prefix position by position, and the toy forward applies the tree mask as Sec. 3.2 states it (a row
sees the committed cache, its own segment causally, and every ancestor segment).
"""
import glob
import inspect
import os
import sys
import types

import pytest

from oracle import jacobi as J
from tests.toy_decode import parse, toy_module

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
VOCAB = 1000


CASES = sorted(glob.glob(os.path.join(GOLDEN, "*.txt")))
CASES = [c for c in CASES if not c.endswith("README.txt")]


@pytest.mark.parametrize("path", CASES, ids=[os.path.basename(c)[:-4] for c in CASES])
def test_decoding_loop_matches_hand_derived_trace(path, monkeypatch):
    spec = parse(path)
    T = spec["prompt"] + spec["truth"]
    monkeypatch.setattr(J, "O", toy_module(T, spec["stationary"]))
    corrupt = spec["corrupt"]

    drawn = set()

    def scripted(seed, pos, it, truth_tok, thr, vocab):
        assert truth_tok == T[pos]
        drawn.add((pos, it))
        return corrupt.get((pos, it), truth_tok)

    monkeypatch.setattr(J, "inject_token", scripted)
    params = J.GenParams(**spec["params"])
    model = types.SimpleNamespace(cfg=types.SimpleNamespace(vocab=VOCAB))
    truth = spec["truth"] if params.init == "inject" else None
    dec = J.JacobiDecoder(model, spec["prompt"], params, truth=truth)
    got = dec.run()
    assert len(got.iters) == len(spec["iters"])
    for i, (rec, want) in enumerate(zip(got.iters, spec["iters"])):
        have = dict(M=rec.M, k=rec.k, winner=rec.winner, k_ra=rec.k_ra, k_cand=list(rec.k_cand),
                    pseudo=list(rec.pseudo), committed=list(rec.committed))
        if "rows" in want:  # the forward's rows: trajectory point, positions, predictions, kinds
            have["rows"] = {k: [int(x) for x in rec.rows[k]] for k in ("tokens", "pos", "pred", "kind")}
        assert have == want, f"iteration {i}"
    assert got.tokens == spec["tokens"]
    # App. C: the trajectory point picked for each block under Eq. 2's schedule
    for w, points in spec.get("noisy", {}).items():
        picks = J.noisy_blocks(got, len(spec["prompt"]), params.block_size, w)
        assert [j for j, _ in picks] == points, f"w = {w}"
    # every scripted corruption was drawn (an entry the loop never asked for is a typo in the script)
    assert set(corrupt) <= drawn


def test_golden_traces_are_lossless():
    """Every trace commits the truth: decoding is lossless whatever the drafts (Sec. 3.2)."""
    for path in CASES:
        spec = parse(path)
        assert spec["tokens"] == spec["truth"][: len(spec["tokens"])], path
        flat = [t for it in spec["iters"] for t in it["committed"]]
        assert flat == spec["truth"][: len(flat)], path            # every committed token is the truth
        assert flat[: len(spec["tokens"])] == spec["tokens"], path  # the output stops inside the last commit


# Plausible mistakes in the decoding loop, each planted (in memory, on the CPU) into a copy of the
# oracle's loop; every one must fail at least one hand-derived trace.
PLANTED = {
    "pseudo-accept compares with the row at the position itself":
        ("blk.q[pk] == main_pred(blk.start + na + pk)", "blk.q[pk] == main_pred(blk.start + na + pk + 1)"),
    "pseudo blocks do not see the blocks before them":
        ("anc = [0] + [(1 << b) - 1 for b in range(1, n_main_seg)]", "anc = [0] * n_main_seg"),
    "candidates ignore the key":
        ("order = [i for i in range(len(self.pool) - 1, -1, -1) if self.pool[i][0] == self.q0]", "order = []"),
    "Jacobi update shifted by one row":
        ("return g[row0 + r]", "return g[row0 + r + 1] if row0 + r + 1 < len(g) else g[row0 + r]"),
    "ties go to the candidate": ("if kc > k:", "if kc >= k:"),
    "pool entries padded with token 0": ("ent += [ent[-1]] * (self.G - len(ent))", "ent += [0] * (self.G - len(ent))"),
    "spawn needs more than ceil(r n)": ("if progress < s:", "if progress <= s:"),
    "promotion keeps the block's own first token": ("draft[0] = self.q0", "pass"),
    "pseudo drafts redrawn with the current iteration":
        ("blk.q = [self._inj(x, self.it + 1) for x in range(lo, hi)]",
         "blk.q = [self._inj(x, self.it) for x in range(lo, hi)]"),
    "spawned block repeats the last committed token":
        ("prev_tok = (last.a + last.q)[-1]", "prev_tok = self._last_committed()"),
    "q0 taken from the draft's rows when a candidate wins":
        ("new_q0, new_q0_margin = g[row0 + k - 1], mg[row0 + k - 1]", "new_q0, new_q0_margin = g[k - 1], mg[k - 1]"),
    "pool entry stops at the end of the real-active draft":
        ("ent = main_tok[k_ra:k_ra + self.G]", "ent = list(ra.q[k_ra:k_ra + self.G])"),
}


@pytest.mark.parametrize("name", sorted(PLANTED))
def test_planted_mistake_fails_a_trace(name, monkeypatch):
    a, b = PLANTED[name]
    src = inspect.getsource(J)
    assert src.count(a) == 1
    mod = types.ModuleType("oracle.jacobi_planted")
    mod.__package__ = "oracle"
    monkeypatch.setitem(sys.modules, mod.__name__, mod)  # its dataclasses look their module up there
    exec(compile(src.replace(a, b), J.__file__, "exec"), mod.__dict__)
    monkeypatch.setattr(sys.modules[__name__], "J", mod)
    caught = 0
    for path in CASES:
        with pytest.MonkeyPatch.context() as mp:
            try:
                test_decoding_loop_matches_hand_derived_trace(path, mp)
            except AssertionError:
                caught += 1
    assert caught > 0, name
