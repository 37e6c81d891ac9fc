"""The CUDA decoding state machine (csrc/jf_decode.cu: verification, pool, pseudo-accept, tail update,
spawn / promote, next rows and chains; Algorithm 1, Sec. 3.2, Eq. 3-4) compiled for the CPU and
checked without a GPU (tests/decode_host/build.py says how the kernels become host code).

* Against the hand-derived traces of tests/golden/ (toy predictor, scripted drafts).
* Its draft-injection rule against the oracle's, on many (seed, position, iteration) keys.
* Against the oracle's decoding loop under the same toy predictor on randomised configurations
  (blocks, spawn ratio, pool, candidates, n-gram length, window mode, batch, injection rate,
  EOS): rows, committed counts, winners and tokens of every iteration must agree.
"""
import ctypes
import glob
import math
import os
import shutil
import types

import numpy as np
import pytest

from oracle import jacobi as J
from tests.toy_decode import chain_predictions, parse, toy_module, wrong_const

pytestmark = pytest.mark.skipif(shutil.which("g++") is None, reason="needs g++")

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
CASES = [c for c in sorted(glob.glob(os.path.join(GOLDEN, "*.txt"))) if not c.endswith("README.txt")]


@pytest.fixture(scope="module")
def hd():
    from tests.decode_host import build as HB

    return HB.load()


def _p(a):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int))


_LAST_TRAJ_ROWS = [0]


def _traj_rows(hd):
    """Rows per record of the trajectory buffer of the last run_device call."""
    return _LAST_TRAJ_ROWS[0]


def run_device(hd, pr, prompts, truths, stationary, V, script=None, wrong=wrong_const, traj_out=None, seq_n=None,
               join=None, chunk=4):
    """Drive the host-compiled state machine with toy predictions. Returns per sequence the list of
    its decoding iterations (rows M, committed count k, winner, output tokens) and its generated
    tokens. traj_out (a list): the trajectory record is switched on and its iterations appended there.
    seq_n: per-sequence block sizes (pr.block_size is then the largest); join: per-sequence join
    iteration (0 = prefilled before the first iteration, else prefilled in `chunk`-row pieces inside
    the iterations)."""
    ns = len(prompts)
    if pr.mode == "ar":
        n, K, mode, pool, C = 1, 1, 1, 0, 0
        seq_n = None
    else:
        n, K, mode, pool = pr.block_size, pr.n_blocks, (1 if pr.mode == "window" else 0), pr.pool_size
        C = pr.cand_per_iter if pool > 0 else 0
    seq_n = list(seq_n) if seq_n is not None else [n] * ns
    join = list(join) if join is not None else [0] * ns
    G = pr.ngram_len or n
    init = 1 if pr.init == "inject" else 0
    s_spawn = math.ceil(pr.spawn_ratio * n - 1e-12)
    T = int(float(np.float32(pr.inject_p)) * 2**53)
    truth_len = min(len(t) - len(p) for t, p in zip(truths, prompts)) if init else 0
    assert not init or truth_len >= pr.max_new + K * n + G + 1
    truth_arr = np.zeros((ns, max(truth_len, 1)), dtype=np.int32)
    for b in range(ns):
        if init:
            truth_arr[b] = truths[b][len(prompts[b]):len(prompts[b]) + truth_len]
    max_rows = ns * max(K * n + C * G, chunk)
    max_chains = ns * (1 + C)
    max_ctx = max(len(p) for p in prompts) + pr.max_new + K * n + G + 8
    sn = np.array(seq_n, dtype=np.int32)
    ss = np.array([math.ceil(pr.spawn_ratio * x - 1e-12) for x in seq_n], dtype=np.int32)
    jn = np.array(join, dtype=np.int32)
    flat = np.array([t for p in prompts for t in p], dtype=np.int32)
    plens = np.array([len(p) for p in prompts], dtype=np.int32)
    assert hd.hd_setup(n, K, s_spawn, pool, G, C, mode, init, T, pr.seed, pr.max_new, pr.eos_id, V, ns,
                       _p(truth_arr), truth_len, max_rows, max_chains, max_ctx, _p(sn), _p(ss), _p(jn), _p(flat),
                       _p(plens), chunk) == 0
    traj_cap = 4 * (pr.max_new + 4)
    if traj_out is not None:
        hd.hd_traj(traj_cap, max_rows)
        _LAST_TRAJ_ROWS[0] = max_rows
    if script is None:
        hd.hd_script(-1, None, None, None)
    else:
        ks = sorted(script)
        cols = [np.array(c, dtype=np.int32) for c in ([k[0] for k in ks], [k[1] for k in ks], [script[k] for k in ks])]
        hd.hd_script(len(ks), *[_p(c) for c in cols])
    committed = [list(p) if join[b] == 0 else [] for b, p in enumerate(prompts)]
    q0 = np.array([truths[b][len(prompts[b])] for b in range(ns)], dtype=np.int32)  # the toy's prefill argmax
    seq_len = np.array([len(p) for p in prompts], dtype=np.int32)
    plast = np.array([p[-1] for p in prompts], dtype=np.int32)
    hd.hd_init(_p(q0), _p(seq_len), _p(plast))
    tok = np.zeros(max_rows, dtype=np.int32)
    pos = np.zeros(max_rows, dtype=np.int32)
    ch = np.zeros((max_chains, 4), dtype=np.int32)
    hdr = np.zeros(4, dtype=np.int32)
    k, win, nout, P = (np.zeros(ns, dtype=np.int32) for _ in range(4))
    cm = np.zeros((ns, 3), dtype=np.int32)
    out = np.zeros((ns, pr.max_new), dtype=np.int32)
    recs = [[] for _ in range(ns)]

    def view():
        hd.hd_view(_p(tok), _p(pos), _p(ch), _p(hdr), _p(k), _p(win), _p(nout), _p(P), _p(cm))
        assert hdr[3] == 0, f"device error word {hdr[3]}"

    view()
    done = [False] * ns
    for _ in range(4 * (pr.max_new + 4)):
        if hdr[2]:
            break
        M = int(hdr[0])
        chains = [tuple(int(v) for v in ch[c]) for c in range(int(hdr[1]))]
        rows = [0] * ns
        for s, _, nr, _ in chains:
            rows[s] += nr
        cur_tok = [int(t) for t in tok[:M]]
        cur_pos = [int(x) for x in pos[:M]]
        pred = np.array(chain_predictions(cur_tok, cur_pos, chains, committed, truths, stationary, wrong),
                        dtype=np.int32)
        fwd = [[] for _ in range(ns)]  # per sequence: its chains' (tokens, positions) in order
        for s_, r0, nr, _ in chains:
            fwd[s_].append((cur_tok[r0:r0 + nr], cur_pos[r0:r0 + nr]))
        prev_out = nout.copy()
        hd.hd_accept(_p(pred), M)
        view()
        hd.hd_out_tokens(_p(out))
        for b in range(ns):
            if done[b]:
                assert k[b] == 0 and rows[b] == 0
                continue
            row0, kk, p_at = (int(v) for v in cm[b])
            assert p_at == len(committed[b])
            if len(committed[b]) < len(prompts[b]) or k[b] == 0:
                # waiting to join, or a prefill chunk: all its rows are committed, nothing is decoded
                assert k[b] == 0 and kk == rows[b] and nout[b] == 0
                committed[b] += cur_tok[row0:row0 + kk]
                assert committed[b] == list(prompts[b][:len(committed[b])])
                continue
            assert kk == k[b]
            committed[b] += cur_tok[row0:row0 + kk]  # the rows the KV commit copies into the cache
            recs[b].append(dict(M=rows[b], k=int(k[b]), winner=int(win[b]),
                                out=[int(t) for t in out[b, prev_out[b]:nout[b]]], fwd=fwd[b]))
            done[b] = bool(nout[b] >= pr.max_new or (pr.eos_id >= 0 and pr.eos_id in out[b, :nout[b]]))
    else:
        raise AssertionError("decoding did not terminate")
    assert all(done)
    if traj_out is not None:
        buf = np.zeros(traj_cap * (2 + 5 * max_rows), dtype=np.int32)
        n_rec = hd.hd_traj_view(_p(buf))
        from paper_2512_14681_gb300.jacobi import trajectory_records

        traj_out += trajectory_records(buf, min(n_rec, traj_cap), max_rows)
    return recs, [[int(t) for t in out[b, :nout[b]]] for b in range(ns)]


def run_oracle(pr, prompt, truth_seq, stationary, V, monkeypatch, wrong=wrong_const, calls=None):
    toy = toy_module(truth_seq, stationary, wrong)
    toy.sm64 = J.O.sm64  # the injection rule's generator stays the oracle's own
    if calls is not None:
        inner = toy.forward

        def forward(model, cache, tokens, pos, seg=None, anc=None, **kw):
            calls.append(([int(t) for t in tokens], [int(x) for x in pos],
                          [0] * len(tokens) if seg is None else [int(v) for v in seg],
                          None if anc is None else [int(v) for v in anc]))
            return inner(model, cache, tokens, pos, seg, anc, **kw)

        toy.forward = forward
    monkeypatch.setattr(J, "O", toy)
    model = types.SimpleNamespace(cfg=types.SimpleNamespace(vocab=V))
    truth = truth_seq[len(prompt):] if pr.init == "inject" else None
    return J.JacobiDecoder(model, prompt, pr, truth=truth).run()


def _tree_equals_chains(tokens, pos, seg, anc):
    """The paper's tree mask (a row sees its own segment causally and every ancestor segment) and the
    kernels' chain rule (a row sees the rows of its chain at positions up to its own) give the same
    visible in-flight rows for this forward."""
    M = len(tokens)
    anc = anc or [0] * (max(seg) + 1)
    chains = _segments(tokens, pos, seg)
    chain_of, start = [], 0
    for ci, (t, _) in enumerate(chains):
        chain_of += [ci] * len(t)
    for i in range(M):
        for j in range(M):
            tree = (seg[j] == seg[i] and pos[j] <= pos[i]) or (seg[j] != seg[i] and (anc[seg[i]] >> seg[j]) & 1)
            chain = chain_of[j] == chain_of[i] and pos[j] <= pos[i]
            if bool(tree) != chain:
                return False
    return True


def _segments(tokens, pos, seg):
    """The oracle's rows of one forward as the kernels' chains: the real-active block with its pseudo
    blocks (segments 0 .. n_main-1, consecutive positions), then one chain per candidate."""
    n_main = 0
    while n_main < len(seg) and (n_main == 0 or seg[n_main] >= seg[n_main - 1]) and \
            (n_main == 0 or pos[n_main] == pos[n_main - 1] + 1):
        n_main += 1
    out = [(tokens[:n_main], pos[:n_main])]
    i = n_main
    while i < len(seg):
        j = i
        while j < len(seg) and seg[j] == seg[i]:
            j += 1
        out.append((tokens[i:j], pos[i:j]))
        i = j
    return out


@pytest.mark.parametrize("path", CASES, ids=[os.path.basename(c)[:-4] for c in CASES])
def test_device_state_machine_matches_hand_derived_trace(hd, path):
    spec = parse(path)
    pr = J.GenParams(**spec["params"])
    T = spec["prompt"] + spec["truth"]
    recs, toks = run_device(hd, pr, [spec["prompt"]], [T], [spec["stationary"]], 1000, script=spec["corrupt"])
    assert len(recs[0]) == len(spec["iters"])
    n_out = 0
    for i, (have, want) in enumerate(zip(recs[0], spec["iters"])):
        # the kernels' output of an iteration: its committed tokens up to max_new or EOS
        out = []
        for t in want["committed"]:
            if n_out >= pr.max_new or (out and out[-1] == pr.eos_id):
                break
            out.append(t)
            n_out += 1
        assert (have["M"], have["k"], have["winner"], have["out"]) == \
            (want["M"], want["k"], want["winner"], out), f"iteration {i}"
    assert toks[0] == spec["tokens"]


def test_device_injection_rule_equals_oracle(hd):
    """The kernels' injection rule and the oracle's, each written from the SplitMix64 definition."""
    rng = np.random.default_rng(5)
    for _ in range(3000):
        seed = int(rng.integers(0, 2**63))
        p = float(rng.choice([0.0, 0.1, 0.3, 0.5, 0.7, 1.0]))
        T = J.inject_threshold(p)
        V = int(rng.choice([2, 3, 1000, 152064]))
        truth_tok = int(rng.integers(0, V))
        x, it = int(rng.integers(0, 1 << 20)), int(rng.integers(0, 4096))
        assert hd.hd_inject_rule(seed, T, V, truth_tok, x, it) == J.inject_token(seed, x, it, truth_tok, T, V)


def _random_case(rng):
    mode = str(rng.choice(["block", "block", "block", "window", "ar"]))
    n = int(rng.choice([1, 2, 3, 4, 6, 8]))
    K = int(rng.integers(1, 4)) if mode == "block" else 1
    pool = int(rng.choice([0, 0, 2, 4, 8]))
    C = int(rng.integers(1, 4)) if pool else 0
    G = int(rng.choice([0, 0, 2, 3, 5]))
    init = str(rng.choice(["repeat", "inject"]))
    return J.GenParams(block_size=n, n_blocks=K, spawn_ratio=float(rng.choice([0.0, 0.25, 0.5, 0.85, 1.0])),
                       pool_size=pool, ngram_len=G, cand_per_iter=C, mode=mode, init=init,
                       inject_p=float(rng.choice([0.0, 0.2, 0.5, 0.9])), seed=int(rng.integers(0, 1 << 30)),
                       max_new=int(rng.integers(1, 40)), eos_id=-1)


@pytest.mark.parametrize("case_seed", range(300))
def test_device_state_machine_equals_oracle_loop(hd, case_seed, monkeypatch):
    """Randomised configurations; a small vocabulary makes chance matches (lucky drafts, pool keys,
    wrong predictions that agree) frequent, so rarely reached branches run."""
    rng = np.random.default_rng(1000 + case_seed)
    pr = _random_case(rng)
    V = int(rng.choice([6, 12, 50]))
    ns = int(rng.integers(1, 4))
    eos = int(rng.integers(2, V)) if rng.random() < 0.25 else -1
    pr = J.GenParams(**{**pr.__dict__, "eos_id": eos})
    prompts, truths, stationary = [], [], []
    for b in range(ns):
        P0 = int(rng.integers(1, 6))
        length = P0 + pr.max_new + pr.n_blocks * pr.block_size + (pr.ngram_len or pr.block_size) + 8
        T = [int(t) for t in rng.integers(2, V, size=length)]
        prompts.append(T[:P0])
        truths.append(T)
        stationary.append({int(x) for x in rng.integers(0, length, size=int(rng.integers(0, length // 3 + 1)))})
    shift = int(rng.integers(0, V))

    def wrong(x, t):
        return (3 * t + x + shift) % V

    traj = []
    recs, toks = run_device(hd, pr, prompts, truths, stationary, V, wrong=wrong, traj_out=traj)
    for b in range(ns):
        calls = []
        want = run_oracle(pr, prompts[b], truths[b], stationary[b], V, monkeypatch, wrong, calls)
        assert toks[b] == want.tokens, f"sequence {b}: {pr}"
        assert len(recs[b]) == len(want.iters), f"sequence {b}: {pr}"
        fwds = calls[1:]  # the first call is the prefill
        for i, (have, it) in enumerate(zip(recs[b], want.iters)):
            assert (have["M"], have["k"], have["winner"]) == (it.M, it.k, it.winner), f"seq {b} iteration {i}: {pr}"
            assert have["fwd"] == _segments(*fwds[i][:3]), f"seq {b} iteration {i}: rows of the forward differ: {pr}"
            assert _tree_equals_chains(*fwds[i]), f"seq {b} iteration {i}: tree mask != chains: {pr}"
            # the trajectory record of this iteration: this sequence's rows, as the oracle's loop built them
            tr = traj[i]
            mine = tr["seq"] == b
            got = {k: [int(v) for v in tr[src][mine]] for k, src in
                   (("tokens", "token"), ("pos", "pos"), ("pred", "pred"), ("kind", "kind"))}
            assert got == {k: [int(v) for v in it.rows[k]] for k in got}, f"seq {b} iteration {i}: trajectory: {pr}"
    # every recorded row belongs to a live sequence, and the record holds one entry per iteration
    assert len(traj) == max(len(r) for r in recs)
    assert all(np.all(t["seq"] >= 0) and t["M"] == int(sum(np.sum(t["seq"] == b) for b in range(ns))) for t in traj)


def test_step_mode_verification(hd):
    """Caller-supplied blocks (the step call): a real-active draft or candidate accepts 1 + the run of
    tokens equal to the prediction of the row before them; a pseudo block, whose rows continue the
    block before it, accepts the run from its first token against the prediction of that block's
    last row; the largest count among the draft and the candidates wins, ties to the earlier block."""
    rng = np.random.default_rng(11)
    for _ in range(2000):
        V = int(rng.integers(2, 5))
        kinds = [0] + [1] * int(rng.integers(0, 3)) + [2] * int(rng.integers(0, 3))
        lens = [int(rng.integers(1, 7)) for _ in kinds]
        M = sum(lens)
        tok = rng.integers(0, V, size=M).astype(np.int32)
        pred = rng.integers(0, V, size=M).astype(np.int32)
        counts = np.zeros(len(kinds), dtype=np.int32)
        out4 = np.zeros(4, dtype=np.int32)
        com = np.full(M, -7, dtype=np.int32)
        kind_a, len_a = np.array(kinds, dtype=np.int32), np.array(lens, dtype=np.int32)
        hd.hd_step(len(kinds), _p(kind_a), _p(len_a), 100, _p(tok), _p(pred), _p(counts), _p(out4), _p(com))
        want, best, win, r0 = [], 0, -1, 0
        for b, (kd, ln) in enumerate(zip(kinds, lens)):
            c = 0 if kd == 1 else 1
            while c < ln and tok[r0 + c] == pred[r0 + c - 1]:
                c += 1
            want.append(c)
            if kd != 1 and c > best:
                best, win, wr0 = c, b, r0
            r0 += ln
        assert list(counts) == want
        assert (out4[0], out4[1], out4[3]) == (win, best, 0)
        assert out4[2] == pred[wr0 + best - 1]
        assert list(com[:best]) == list(tok[wr0:wr0 + best])


@pytest.mark.parametrize("case_seed", range(200))
def test_device_serving_block_sizes_and_late_joins(hd, case_seed, monkeypatch):
    """Serving several sequences at once: each with its own block size, some joining later with their
    prompts prefilled in chunks inside the iterations (beside the running sequences' Jacobi rows).
    Every sequence must decode exactly as the oracle's loop decodes it alone at its own block size:
    the same rows (as chains), committed counts, winners and tokens, iteration by iteration; its
    prefill chunks commit its prompt in order; the trajectory record marks them as prefill rows."""
    rng = np.random.default_rng(5000 + case_seed)
    pr = _random_case(rng)
    if pr.mode == "ar":
        pr = J.GenParams(**{**pr.__dict__, "mode": "block", "block_size": 4})
    V = int(rng.choice([6, 12, 50]))
    ns = int(rng.integers(1, 6))
    seq_n = [int(rng.integers(1, pr.block_size + 1)) for _ in range(ns)]
    join = [int(rng.choice([0, 0, 1, 2, 5, 9])) for _ in range(ns)]
    chunk = int(rng.choice([1, 2, 3, 5, 64]))
    prompts, truths, stationary = [], [], []
    for b in range(ns):
        P0 = int(rng.integers(1, 12))
        length = P0 + pr.max_new + pr.n_blocks * pr.block_size + (pr.ngram_len or pr.block_size) + 8
        T = [int(t) for t in rng.integers(2, V, size=length)]
        prompts.append(T[:P0])
        truths.append(T)
        stationary.append({int(x) for x in rng.integers(0, length, size=int(rng.integers(0, length // 3 + 1)))})
    shift = int(rng.integers(0, V))

    def wrong(x, t):
        return (3 * t + x + shift) % V

    traj = []
    recs, toks = run_device(hd, pr, prompts, truths, stationary, V, wrong=wrong, traj_out=traj, seq_n=seq_n,
                            join=join, chunk=chunk)
    for b in range(ns):
        prb = J.GenParams(**{**pr.__dict__, "block_size": seq_n[b]})
        calls = []
        want = run_oracle(prb, prompts[b], truths[b], stationary[b], V, monkeypatch, wrong, calls)
        assert toks[b] == want.tokens, f"sequence {b}: {prb} join {join[b]}"
        assert len(recs[b]) == len(want.iters), f"sequence {b}: {prb}"
        fwds = calls[1:]
        for i, (have, it) in enumerate(zip(recs[b], want.iters)):
            assert (have["M"], have["k"], have["winner"]) == (it.M, it.k, it.winner), f"seq {b} iteration {i}: {prb}"
            assert have["fwd"] == _segments(*fwds[i][:3]), f"seq {b} iteration {i}: rows differ: {prb}"
        # its records: prefill chunks (kind 3) covering the prompt in order when it joined late, then
        # its decoding iterations, each with the oracle's rows
        mine = [{k: t[k][t["seq"] == b] for k in ("kind", "pos", "token", "pred")} for t in traj]
        mine = [m for m in mine if m["kind"].size]
        pre = [m for m in mine if np.all(m["kind"] == 3)]
        if join[b] > 0:
            assert [int(x) for m in pre for x in m["token"]] == prompts[b]
            assert [int(x) for m in pre for x in m["pos"]] == list(range(len(prompts[b])))
            # its first chunk runs in forward join[b], or earlier only in a forward no other sequence uses
            first = next(i for i, t in enumerate(traj) if np.any((t["seq"] == b) & (t["kind"] == 3)))
            assert first == join[b] or (first < join[b] and np.all(traj[first]["seq"] == b)), (first, join)
        else:
            assert not pre
        dec = [m for m in mine if not np.any(m["kind"] == 3)]
        assert len(dec) == len(want.iters)
        for m, it in zip(dec, want.iters):
            assert [int(x) for x in m["token"]] == list(it.rows["tokens"])
            assert [int(x) for x in m["kind"]] == list(it.rows["kind"])


@pytest.mark.parametrize("case_seed", range(150))
def test_device_training_points_equal_oracle(hd, case_seed, monkeypatch):
    """App. C's training points (Eq. 2 schedule) picked by the kernel from its own trajectory record
    equal the oracle's picks from its decoding loop, for every block of every sequence and several
    window sizes."""
    rng = np.random.default_rng(9000 + case_seed)
    n = int(rng.choice([1, 2, 3, 4, 6, 8]))
    pool = int(rng.choice([0, 0, 4]))
    pr = J.GenParams(block_size=n, n_blocks=1, pool_size=pool, cand_per_iter=(1 if pool else 0),
                     mode="block", init=str(rng.choice(["repeat", "inject"])),
                     inject_p=float(rng.choice([0.2, 0.5, 0.9])), seed=int(rng.integers(0, 1 << 30)),
                     max_new=int(rng.integers(n, 40)), eos_id=-1)
    V = int(rng.choice([6, 12, 50]))
    ns = int(rng.integers(1, 4))
    prompts, truths, stationary = [], [], []
    for b in range(ns):
        P0 = int(rng.integers(1, 6))
        length = P0 + pr.max_new + n + n + 8
        T = [int(t) for t in rng.integers(2, V, size=length)]
        prompts.append(T[:P0])
        truths.append(T)
        stationary.append({int(x) for x in rng.integers(0, length, size=int(rng.integers(0, length // 3 + 1)))})
    shift = int(rng.integers(0, V))

    def wrong(x, t):
        return (3 * t + x + shift) % V

    traj = []
    recs, toks = run_device(hd, pr, prompts, truths, stationary, V, wrong=wrong, traj_out=traj)
    n_rec = len(traj)
    for b in range(ns):
        want = run_oracle(pr, prompts[b], truths[b], stationary[b], V, monkeypatch, wrong)
        assert toks[b] == want.tokens
        fixed = np.array(toks[b], dtype=np.int32)
        nb = len(toks[b]) // n
        for w in (1, 2, 3, 4, 8):
            noisy = np.full((max(nb, 1), n), -9, dtype=np.int32)
            point = np.full(max(nb, 1), -9, dtype=np.int32)
            hd.hd_traj_noisy(n_rec, _traj_rows(hd), b, _p(fixed), len(prompts[b]), n, w, nb, _p(noisy), _p(point))
            picks = J.noisy_blocks(want, len(prompts[b]), n, w)
            # the record holds one entry per forward of all sequences; the oracle counts this sequence's
            # iterations: map the kernel's record index to the sequence's own iteration index
            own = [i for i, t in enumerate(traj) if np.any(t["seq"] == b)]
            to_own = {r: k for k, r in enumerate(own)}
            got = [(to_own.get(int(point[i]), len(want.iters)), [int(x) for x in noisy[i]]) for i in range(nb)]
            assert got == [(j, list(s)) for j, s in picks], f"seq {b} w {w}: {pr}"
