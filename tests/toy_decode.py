"""Scripted toy predictor and the hand-derived trace format (tests/golden/), shared by the tests of
the oracle's decoding loop and of the CUDA state machine compiled for the host.

Toy predictor: T is the true sequence by absolute position. A row holding token t at position x
predicts T[x+1] when t == T[x] and the token it sees at x-1 (committed cache or a visible in-flight
row) equals T[x-1], or when x+1 is a stationary position; otherwise it predicts wrong(x, t). The
predictor stands in for the transformer's greedy argmax; what a row sees follows the tree mask of
Sec. 3.2 (committed cache, its own segment causally, every ancestor segment).
"""
import types

import numpy as np

WRONG = 1


def wrong_const(x, t):
    return WRONG


def toy_predict(T, stationary, x, own, prev, wrong=wrong_const):
    """prev: the visible token at x-1, None if no row at x-1 is visible (x = 0 needs none)."""
    ok = own == T[x] and (x == 0 or (prev is not None and prev == T[x - 1]))
    return T[x + 1] if ok or (x + 1) in stationary else wrong(x, own)


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
        elif head == "rows":
            # the rows of the preceding iteration's forward: tokens, positions, predictions, kinds
            rows = {}
            for item in rest.split():
                k, v = item.split("=")
                rows[k] = _ints(v)
            spec["iters"][-1]["rows"] = rows
        elif head == "noisy":
            # App. C's pick per block for a window size w: noisy w=<w> points=<iteration of each block's point>
            kv = dict(item.split("=") for item in rest.split())
            spec.setdefault("noisy", {})[int(kv["w"])] = _ints(kv["points"])
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


def toy_module(T, stationary, wrong=wrong_const):
    """Stand-in for the oracle module inside its decoding loop: forward() over rows with segment
    ids and ancestor masks, and the cache."""

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
                prev = None
            elif x - 1 < P:
                prev = cache.toks[x - 1]
            else:
                seen = [j for j in range(M) if pos[j] == x - 1 and
                        ((seg[j] == seg[i] and pos[j] <= x) or (seg[j] != seg[i] and (anc[seg[i]] >> seg[j]) & 1))]
                assert len(seen) <= 1, "two visible rows at one position"
                prev = tokens[seen[0]] if seen else None
            pred.append(toy_predict(T, stationary, x, tokens[i], prev, wrong))
        cache.last = (tokens, pos)
        return types.SimpleNamespace(argmax=np.array(pred, dtype=np.int32), margin=np.ones(M))

    return types.SimpleNamespace(forward=forward, Cache=ToyCache)


def chain_predictions(tok, pos, chains, committed, truths, stationary, wrong=wrong_const):
    """Toy predictions for the rows of a forward described by chains (seq, row0, nrows, pos0): a row
    sees its sequence's committed tokens and the rows of its chain at positions up to its own."""
    pred = [None] * len(tok)
    for seq, row0, nrows, pos0 in chains:
        assert pos0 == len(committed[seq]), "chain does not start at the committed length"
        T = truths[seq]
        for r in range(row0, row0 + nrows):
            x = pos[r]
            assert x == pos0 + (r - row0), "chain rows are not at consecutive positions"
            if x - 1 < 0:
                prev = None
            elif x - 1 < pos0:
                prev = committed[seq][x - 1]
            else:
                prev = tok[row0 + (x - 1 - pos0)]
            pred[r] = toy_predict(T, stationary[seq], x, tok[r], prev, wrong)
    assert all(p is not None for p in pred), "a row belongs to no chain"
    return pred
