"""Greedy AR decoding and Jacobi decoding on the CPU oracle (TEST INFRASTRUCTURE ONLY).

Follows Jacobi Forcing (arXiv 2512.14681):
  * greedy AR decoding, Eq. 1;
  * the Jacobi fixed-point update, Eq. 3: one forward with a causal mask updates every
    position of a block from the previous guess; the first position is exact each time;
  * block-sequential generation, Eq. 4; the running-window variant of Sec. 4.2;
  * multi-block decoding and rejection recycling, Sec. 3.2 and Algorithm 1 (Appendix A):
    assemble -> forward -> verify (longest matching prefix, pool candidates for the
    real-active block) -> tail update and pool push -> cache trim -> spawn -> promote.

Conventions where the paper is silent are the readings listed in the design notes:
  * the draft of the real-active (RA) block starts with q0, the token already known to be
    correct (the greedy prediction after the last committed token), so every iteration
    commits k >= 1 tokens: k = 1 + the longest run of draft tokens equal to the prediction
    of the row before them;
  * a pseudo-active block has no free first token: it pseudo-accepts the longest prefix of
    its draft equal to the prediction of the row before each token;
  * the winner among the RA draft and the recycled candidates is the largest k, ties going to
    the RA draft, then to the lower candidate index;
  * the pool keeps the rejected RA tail (padded to the n-gram length with the following
    in-flight tokens, then with its last token), FIFO, keyed by its first token; a candidate
    is [q0] + an entry's other tokens; entries whose key equals q0 rank first, most recent first,
    then the other entries, most recent first;
  * spawn: while fewer than K blocks are active and the newest block has at least ceil(r n)
    accepted tokens, a pseudo block is appended; promote: when the RA block is complete the
    next block becomes RA, its first token replaced by q0, and is verified again;
  * draft tokens that the algorithm leaves free come from the initial-guess rule: "repeat"
    (the last committed token, or for a spawned block the last draft token before it), or
    "inject": the true greedy continuation at that position, replaced with probability p by
    another uniform token, drawn from a counter-based generator keyed by (seed, position,
    iteration). The pure Jacobi update (next draft = this iteration's predictions) applies
    in "repeat" mode.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

from . import oracle as O

TWO53 = 2**53


@dataclass
class GenParams:
    block_size: int = 8          # n
    n_blocks: int = 1            # K
    spawn_ratio: float = 0.0     # r
    pool_size: int = 0           # rejection-recycling pool capacity (0 = off)
    ngram_len: int = 0           # G (0 = n)
    cand_per_iter: int = 0       # recycled candidates verified per iteration
    mode: str = "block"          # "block" | "window" | "ar"
    init: str = "repeat"         # "repeat" | "inject"
    inject_p: float = 0.0
    seed: int = 0
    max_new: int = 64
    eos_id: int = -1


@dataclass
class IterRecord:
    M: int                       # in-flight rows of the forward
    k: int                       # tokens committed
    winner: int                  # 0 = RA draft, c+1 = candidate c
    k_ra: int
    k_cand: list
    pseudo: list                 # pseudo-accepted counts per pseudo block
    committed: list
    # the forward's rows, one entry per row: the Jacobi trajectory point y^(j) of the real-active block
    # (Sec. 2.1), the pseudo blocks after it and the candidates, with their greedy predictions y^(j+1)
    # (kind 0 = real-active, 1 = pseudo-active, 2 = recycled candidate)
    rows: dict = field(default_factory=dict)


@dataclass
class GenResult:
    tokens: list                 # new tokens (exactly max_new unless EOS)
    margins: list                # fp32 top-1 minus top-2 logit of the decision behind each token
    iters: list = field(default_factory=list)

    @property
    def counts(self):
        return [it.k for it in self.iters]


def inject_threshold(p: float) -> int:
    """Corruption threshold T = floor(p32 * 2^53) for the fp32 value p32 of p."""
    return int(float(np.float32(p)) * TWO53)


def inject_token(seed: int, pos: int, it: int, truth_tok: int, T: int, vocab: int) -> int:
    """Draft-injection rule: s = SplitMix64 output `pos` of the stream seeded with `seed`;
    r1, r2 = outputs 2 it and 2 it + 1 of the stream started at s. Corrupt iff
    (r1 >> 11) < T; the replacement is (truth + 1 + r2 mod (V - 1)) mod V != truth."""
    s = O.sm64(seed, pos)
    r1 = O.sm64(s, 2 * it)
    if (r1 >> 11) >= T:
        return truth_tok
    r2 = O.sm64(s, 2 * it + 1)
    return (truth_tok + 1 + r2 % (vocab - 1)) % vocab


def prefill(model: O.Model, cache: O.Cache, prompt):
    """Commit the prompt's KV and return (q0, margin): the greedy next token."""
    prompt = np.asarray(prompt, dtype=np.int32)
    P0 = len(cache)
    n = prompt.size
    out = O.forward(model, cache, prompt, np.arange(P0, P0 + n, dtype=np.int32))
    cache.commit(np.arange(n, dtype=np.int32))
    return int(out.argmax[-1]), float(out.margin[-1])


def generate_ar(model: O.Model, prompt, max_new: int, eos_id: int = -1, max_ctx: int | None = None) -> GenResult:
    """Greedy AR decoding (Eq. 1): one forward per token."""
    prompt = list(prompt)
    cache = O.Cache(model, max_ctx or (len(prompt) + max_new + 1), max(len(prompt), 1))
    q0, mg = prefill(model, cache, prompt)
    toks, margins = [], []
    while True:
        toks.append(q0)
        margins.append(mg)
        if len(toks) >= max_new or q0 == eos_id:
            break
        P = len(cache)
        out = O.forward(model, cache, [q0], [P])
        cache.commit([0])
        q0, mg = int(out.argmax[0]), float(out.margin[0])
    return GenResult(toks, margins)


class _Block:
    def __init__(self, start, a, q):
        self.start = start       # absolute position of the block's first token
        self.a = list(a)         # pseudo-accepted tokens (pseudo blocks only)
        self.q = list(q)         # draft tokens


class JacobiDecoder:
    """One sequence decoded with Jacobi iterations (Eq. 3-4, Algorithm 1)."""

    def __init__(self, model: O.Model, prompt, params: GenParams, truth=None, max_ctx: int | None = None):
        pr = params
        if pr.mode not in ("block", "window", "ar"):
            raise ValueError("mode")
        if pr.init not in ("repeat", "inject"):
            raise ValueError("init")
        if pr.mode == "ar":
            pr = GenParams(**{**pr.__dict__, "block_size": 1, "mode": "window", "n_blocks": 1, "pool_size": 0,
                              "cand_per_iter": 0})
        if pr.n_blocks > 1 and pr.mode != "block":
            raise ValueError("multi-block decoding needs block mode")
        self.p = pr
        self.model = model
        self.V = model.cfg.vocab
        self.n = pr.block_size
        self.G = pr.ngram_len or pr.block_size
        self.prompt = [int(t) for t in prompt]
        self.P0 = len(self.prompt)
        if pr.init == "inject":
            need = pr.max_new + pr.n_blocks * self.n + self.G + 1
            if truth is None or len(truth) < need:
                raise ValueError(f"inject mode needs a truth continuation of >= {need} tokens")
        self.truth = None if truth is None else [int(t) for t in truth]
        self.T = inject_threshold(pr.inject_p)
        rows_cap = pr.n_blocks * self.n + max(pr.cand_per_iter, 0) * self.G + 1
        self.cache = O.Cache(model, max_ctx or (self.P0 + pr.max_new + pr.n_blocks * self.n + self.G + 2),
                             max(self.P0, rows_cap))
        self.q0, self.q0_margin = prefill(model, self.cache, self.prompt)
        self.P = len(self.cache)
        self.it = 0
        self.tokens: list = []
        self.margins: list = []
        self.iters: list = []
        self.pool: list = []     # FIFO of n-grams, oldest first
        self.done = False
        self.blocks = [_Block(self.P, [], [self.q0] + self._fill(self.P + 1, self.P + self._win(), self.it))]
        self._spawn(self.it)
        self.cands = []

    # -- initial guesses ---------------------------------------------------------------
    def _win(self):
        return self.n

    def _last_committed(self):
        return self.tokens[-1] if self.tokens else self.prompt[-1]

    def _inj(self, pos, it):
        return inject_token(self.p.seed, pos, it, self.truth[pos - self.P0], self.T, self.V)

    def _fill(self, lo, hi, it, repeat_tok=None):
        """Draft tokens for positions lo..hi-1 from the initial-guess rule."""
        if self.p.init == "inject":
            return [self._inj(x, it) for x in range(lo, hi)]
        t = self._last_committed() if repeat_tok is None else repeat_tok
        return [t] * max(0, hi - lo)

    def _spawn(self, it):
        if self.p.n_blocks <= 1:
            return
        s = math.ceil(self.p.spawn_ratio * self.n)
        while len(self.blocks) < self.p.n_blocks:
            last = self.blocks[-1]
            progress = (self.P - last.start) if last is self.blocks[0] else len(last.a)
            if progress < s:
                break
            start = last.start + self.n
            prev_tok = (last.a + last.q)[-1]
            self.blocks.append(_Block(start, [], self._fill(start, start + self.n, it, repeat_tok=prev_tok)))

    # -- one iteration (Algorithm 1 loop body) ------------------------------------------
    def step(self) -> IterRecord:
        P, n = self.P, self.n
        ra = self.blocks[0]
        # assemble: main chain (RA draft, then a_b || q_b of each pseudo block), then candidates
        main_tok = list(ra.q)
        seg_main = [0] * len(ra.q)
        for b, blk in enumerate(self.blocks[1:], start=1):
            main_tok += blk.a + blk.q
            seg_main += [b] * n
        n_main_seg = len(self.blocks)
        tokens = list(main_tok)
        pos = list(range(P, P + len(main_tok)))
        seg = list(seg_main)
        anc = [0] + [(1 << b) - 1 for b in range(1, n_main_seg)]
        cand_rows = []
        for c, ctoks in enumerate(self.cands):
            sid = n_main_seg + c
            cand_rows.append(len(tokens))
            tokens += ctoks
            pos += list(range(P, P + len(ctoks)))
            seg += [sid] * len(ctoks)
            anc.append(0)
        out = O.forward(self.model, self.cache, tokens, pos, seg, anc)
        g = [int(x) for x in out.argmax]
        mg = [float(x) for x in out.margin]

        # verification of the RA draft and of each candidate (greedy rejection sampling)
        def lead(draft, row0):
            k = 1
            while k < len(draft) and draft[k] == g[row0 + k - 1]:
                k += 1
            return k

        L = len(ra.q)
        k_ra = lead(ra.q, 0)
        k_c = [lead(ct, r0) for ct, r0 in zip(self.cands, cand_rows)]
        winner, k, row0, wtoks = 0, k_ra, 0, ra.q
        for c, kc in enumerate(k_c):
            if kc > k:
                winner, k, row0, wtoks = c + 1, kc, cand_rows[c], self.cands[c]
        committed = list(wtoks[:k])
        cmargins = [self.q0_margin] + [mg[row0 + i - 1] for i in range(1, k)]
        new_q0, new_q0_margin = g[row0 + k - 1], mg[row0 + k - 1]
        # cache trim: only the winner's first k rows become cache entries
        self.cache.commit(list(range(row0, row0 + k)))
        self.P = P + k

        # pseudo-active blocks: pseudo-accept against the main chain's predictions
        pseudo_counts = []
        main_end = P + len(main_tok)

        def main_pred(x):           # prediction for position x from the main chain (row at x-1)
            return g[x - 1 - P]

        for blk in self.blocks[1:]:
            na = len(blk.a)
            pk = 0
            while pk < len(blk.q) and blk.q[pk] == main_pred(blk.start + na + pk):
                pk += 1
            pseudo_counts.append(pk)
            blk.a += blk.q[:pk]
            lo = blk.start + len(blk.a)
            hi = blk.start + n
            if self.p.init == "inject":
                blk.q = [self._inj(x, self.it + 1) for x in range(lo, hi)]
            else:
                blk.q = [main_pred(x) for x in range(lo, hi)]

        # rejection recycling: push the rejected RA tail
        if self.p.pool_size > 0 and k_ra < L:
            ent = main_tok[k_ra:k_ra + self.G]
            ent += [ent[-1]] * (self.G - len(ent))
            self.pool.append(ent)
            if len(self.pool) > self.p.pool_size:
                self.pool.pop(0)

        # bookkeeping of committed tokens (EOS / max_new)
        for t, m_ in zip(committed, cmargins):
            if self.done:
                break
            self.tokens.append(t)
            self.margins.append(m_)
            if len(self.tokens) >= self.p.max_new or t == self.p.eos_id:
                self.done = True
        self.q0, self.q0_margin = new_q0, new_q0_margin
        nit = self.it + 1

        def tail_pred(x):           # prediction for position x: winner chain row if present, else main chain
            r = x - 1 - P
            wlen = len(wtoks)
            if 0 <= r < wlen:
                return g[row0 + r]
            if x - 1 < main_end:
                return main_pred(x)
            return None

        # RA tail update / block completion / promotion
        if self.p.mode == "window":
            tail = []
            for x in range(self.P + 1, self.P + n):
                if self.p.init == "inject":
                    tail.append(self._inj(x, nit))
                else:
                    t = tail_pred(x)
                    tail.append(self._last_committed() if t is None else t)
            self.blocks[0] = _Block(self.P, [], [self.q0] + tail)
        elif self.P >= ra.start + n:
            if len(self.blocks) > 1:
                nb = self.blocks[1]
                draft = nb.a + nb.q
                draft[0] = self.q0
                self.blocks = [_Block(nb.start, [], draft)] + self.blocks[2:]
            else:
                self.blocks[0] = _Block(self.P, [], [self.q0] + self._fill(self.P + 1, self.P + n, nit))
        else:
            hi = ra.start + n
            if self.p.init == "inject":
                tail = [self._inj(x, nit) for x in range(self.P + 1, hi)]
            else:
                tail = [tail_pred(x) for x in range(self.P + 1, hi)]
            self.blocks[0] = _Block(ra.start, [], [self.q0] + tail)
        self._spawn(nit)

        # candidates for the next iteration
        self.cands = []
        if self.p.pool_size > 0 and self.p.cand_per_iter > 0:
            Ln = len(self.blocks[0].q)
            if Ln >= 2:
                order = [i for i in range(len(self.pool) - 1, -1, -1) if self.pool[i][0] == self.q0]
                order += [i for i in range(len(self.pool) - 1, -1, -1) if self.pool[i][0] != self.q0]
                for i in order[:self.p.cand_per_iter]:
                    ent = self.pool[i]
                    self.cands.append(([self.q0] + ent[1:])[:Ln])
        kinds = [0] * len(ra.q) + [1] * (len(main_tok) - len(ra.q)) + [2] * (len(tokens) - len(main_tok))
        rec = IterRecord(len(tokens), k, winner, k_ra, k_c, pseudo_counts, committed,
                         dict(tokens=list(tokens), pos=list(pos), pred=g, kind=kinds, margin=mg))
        self.iters.append(rec)
        self.it = nit
        return rec

    def run(self) -> GenResult:
        while not self.done:
            self.step()
        return GenResult(self.tokens[: self.p.max_new], self.margins[: self.p.max_new], self.iters)


def generate_jacobi(model: O.Model, prompt, params: GenParams, truth=None, max_ctx=None) -> GenResult:
    return JacobiDecoder(model, prompt, params, truth=truth, max_ctx=max_ctx).run()


# ------------------------------------------------------------------------------------------
# Training data from Jacobi trajectories (Sec. 3.1, Eq. 2; App. C)
# ------------------------------------------------------------------------------------------
def noise_ratio(i: int, w: int):
    """Eq. 2: the linear progressive schedule over windows of w blocks, W = {0, 1/w, ..., (w-1)/w},
    t_i = W[i mod w], as the exact fraction (i mod w, w). Blocks are counted from 0, so that the ratio
    rises from 0 within each window as the text states."""
    return i % w, w


def block_points(result: GenResult, P0: int, n: int, block: int):
    """The Jacobi trajectory of block `block` (positions P0 + block*n .. + n - 1) of a single-block,
    block-mode run: one point per iteration whose real-active rows lie in the block -- the block's n
    tokens at that iteration, i.e. the committed tokens before the draft (the fixed point there) and the
    draft tokens from the first draft position on -- and finally the fixed point itself (Sec. 2.1)."""
    fixed = [int(t) for t in result.tokens]
    b0 = P0 + block * n
    pts = []
    for j, it in enumerate(result.iters):
        ra = [(p, t) for p, t, k in zip(it.rows["pos"], it.rows["tokens"], it.rows["kind"]) if k == 0]
        if not ra or not (b0 <= ra[0][0] < b0 + n):
            continue
        state = [fixed[x - P0] for x in range(b0, b0 + n)]
        for p, t in ra:
            if b0 <= p < b0 + n:
                state[p - b0] = int(t)
        pts.append((j, state))
    pts.append((len(result.iters), [fixed[x - P0] for x in range(b0, b0 + n)]))
    return pts


def noisy_blocks(result: GenResult, P0: int, n: int, w: int):
    """App. C: for every full block i of the generation, the point of its Jacobi trajectory whose
    fraction of unconverged tokens (positions that differ from the fixed point, over n) is closest to
    t_i of Eq. 2; on a tie the earlier point. Returns [(point index, n tokens)] per block, the index
    being the iteration of the point's forward (len(result.iters) for the fixed point)."""
    fixed = [int(t) for t in result.tokens]
    out = []
    for i in range(len(fixed) // n):
        a, b = noise_ratio(i, w)
        clean = fixed[i * n:(i + 1) * n]
        best = None
        for j, state in block_points(result, P0, n, i):
            noisy = sum(1 for x, y in zip(state, clean) if x != y)
            dist = abs(noisy * b - a * n)  # |noisy / n - a / b| scaled by n * b
            if best is None or dist < best[0]:
                best = (dist, j, state)
        out.append((best[1], best[2]))
    return out
