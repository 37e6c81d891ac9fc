"""The oracle's decoding loop (Algorithm 1, Sec. 3.2; Eq. 3-4) against hand-derived traces (no GPU).

The transformer is replaced by a scripted toy predictor (described in tests/golden/README.txt) and the
draft injection by a scripted corruption list, so that every iteration's rows, accepted counts,
pseudo-accepted counts, winner and committed tokens can be worked out by hand. The traces under
tests/golden/ were derived that way from the rules; this test runs the oracle's loop on the same
scripts and compares iteration by iteration. The toy cache checks that the committed rows extend the
prefix position by position, and the toy forward applies the tree mask as Sec. 3.2 states it (a row
sees the committed cache, its own segment causally, and every ancestor segment).
"""
import glob
import os
import types

import numpy as np
import pytest

from oracle import jacobi as J

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
WRONG = 1
VOCAB = 1000


def _ints(s):
    return [int(t) for t in s.replace(",", " ").split()] if s.strip() else []


def parse(path):
    spec = {"iters": [], "corrupt": {}, "stationary": set()}
    for raw in open(path):
        line = raw.split("#", 1)[0].strip()
        if not line:
            continue
        head, _, rest = line.partition(" ")
        if head == "params":
            kw = {}
            for item in rest.split():
                k, v = item.split("=")
                kw[k] = v if k in ("mode", "init") else (float(v) if k == "spawn_ratio" else int(v))
            spec["params"] = kw
        elif head == "model":
            k, _, v = rest.partition("=")
            assert k == "stationary"
            spec["stationary"] = set(_ints(v))
        elif head in ("prompt", "truth", "tokens"):
            spec[head] = _ints(rest)
        elif head == "corrupt":
            for item in rest.split():
                at, tok = item.split("=")
                pos, it = at.split("@")
                spec["corrupt"][(int(pos), int(it))] = int(tok)
        elif head == "iter":
            rec = {}
            for item in rest.split():
                k, v = item.split("=")
                rec[k] = _ints(v) if k in ("k_cand", "pseudo", "committed") else int(v)
            spec["iters"].append(rec)
        else:
            raise ValueError(f"{path}: unknown line {line!r}")
    return spec


class ToyCache:
    """Committed tokens of one sequence; commit() takes rows of the last forward, in order, and checks
    that they extend the prefix position by position (the cache trim of Algorithm 1)."""

    def __init__(self, model, max_ctx, max_rows):
        self.toks = []
        self.last = None

    def __len__(self):
        return len(self.toks)

    def commit(self, rows):
        tokens, pos = self.last
        for r in list(rows):
            assert pos[r] == len(self.toks), "committed row is not the next position"
            self.toks.append(int(tokens[r]))


def toy_module(T, stationary):
    def forward(model, cache, tokens, pos, seg=None, anc=None, **_):
        tokens = [int(t) for t in tokens]
        pos = [int(p) for p in pos]
        M = len(tokens)
        seg = [0] * M if seg is None else [int(s) for s in seg]
        anc = [0] * (max(seg) + 1) if anc is None else [int(a) for a in anc]
        P = len(cache)
        assert all(p >= P for p in pos), "an in-flight row overlaps the committed prefix"
        pred = []
        for i in range(M):
            x = pos[i]
            if x - 1 < 0:
                prev_ok = True
            elif x - 1 < P:
                prev_ok = cache.toks[x - 1] == T[x - 1]
            else:
                seen = [j for j in range(M) if pos[j] == x - 1 and
                        ((seg[j] == seg[i] and pos[j] <= x) or (seg[j] != seg[i] and (anc[seg[i]] >> seg[j]) & 1))]
                assert len(seen) <= 1, "two visible rows at one position"
                prev_ok = bool(seen) and tokens[seen[0]] == T[x - 1]
            ok = tokens[i] == T[x] and prev_ok
            pred.append(T[x + 1] if ok or (x + 1) in stationary else WRONG)
        cache.last = (tokens, pos)
        return types.SimpleNamespace(argmax=np.array(pred, dtype=np.int32), margin=np.ones(M))

    return types.SimpleNamespace(forward=forward, Cache=ToyCache)


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
        assert have == want, f"iteration {i}"
    assert got.tokens == spec["tokens"]
    # every scripted corruption was drawn (an entry the loop never asked for is a typo in the script)
    assert set(corrupt) <= drawn


def test_golden_traces_are_lossless():
    """Every trace commits the truth: decoding is lossless whatever the drafts (Sec. 3.2)."""
    for path in CASES:
        spec = parse(path)
        assert spec["tokens"] == spec["truth"][: len(spec["tokens"])], path
        flat = [t for it in spec["iters"] for t in it["committed"]]
        assert flat == spec["tokens"], path
