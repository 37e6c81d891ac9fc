"""Helpers shared by the GPU parity tests (no arithmetic of the method)."""
from __future__ import annotations

import numpy as np
import pytest

# Logit tolerances of the comparison (max-abs): fp32 models 1e-4, bf16 models 3e-2. A greedy
# decision may legitimately differ only where the oracle's top-1/top-2 margin is below twice
# the tolerance; such positions are flagged and listed instead of failing.
LOGIT_TOL = {False: 1e-4, True: 3e-2}


def flag_tol(bf16: bool) -> float:
    return 2 * LOGIT_TOL[bf16]


def noise_floor(case: str) -> dict:
    """The oracle's own logit spread under a one-fp32-unit perturbation at every bf16 rounding point
    for one of the wide forwards (tests/golden/logit_noise_floor.json, written by the script beside
    it from the oracle alone): {"max_abs", "std"}."""
    import json
    import os

    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "logit_noise_floor.json")
    return json.load(open(path))["cases"][case]


def wide_logit_tol(case: str) -> tuple:
    """(max-abs, std) bounds of a wide bf16 forward's logits against the oracle: the fixed 3e-2 bound,
    or twice what fp32 accumulation alone spreads the oracle's logits by, whichever is larger; and
    twice the oracle's own spread for the standard deviation of the differences."""
    f = noise_floor(case)
    return max(LOGIT_TOL[True], 2 * f["max_abs"]), 2 * f["std"]


def need_gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch


def _first_row_tie(ref, bf16: bool):
    """First iteration of the oracle's run whose forward had a row at a near-tie (top-1/top-2 margin
    below twice the tolerance): from there on the two runs' drafts, and so their counts, may part
    even while their committed tokens agree. None if the record has no such row (or no rows)."""
    for i, it in enumerate(getattr(ref, "iters", []) or []):
        rows = getattr(it, "rows", None)
        if rows and "margin" in rows and len(rows["margin"]) and min(rows["margin"]) < flag_tol(bf16):
            return i
    return None


def compare_generation(gpu_tokens, gpu_counts, ref, bf16: bool, report=None):
    """Token sequences must match exactly up to the first divergence, which must sit at a
    flagged near-tie of the oracle; per-iteration counts must match for every iteration that
    ends before it, except from an iteration whose forward (or an earlier one) had a row at a
    near-tie of the oracle, where the drafts may part (flagged too). Returns the flagged position
    (tokens decided before the point where the runs may part) or None."""
    gpu_tokens = [int(t) for t in gpu_tokens]
    div = None
    for i, (a, b) in enumerate(zip(gpu_tokens, ref.tokens)):
        if a != b:
            div = i
            break
    if div is not None:
        m = ref.margins[div]
        assert m < flag_tol(bf16), f"token {div}: gpu {gpu_tokens[div]} vs oracle {ref.tokens[div]}, margin {m}"
        if report is not None:
            report.append(("flagged", div, m))
    else:
        assert len(gpu_tokens) == len(ref.tokens)
    done = 0
    gc = [int(k) for k in gpu_counts]
    tie_it = _first_row_tie(ref, bf16)
    for it, (kg, ko) in enumerate(zip(gc, ref.counts)):
        if div is not None and done + ko >= div:
            break
        if kg != ko and tie_it is not None and it >= tie_it:
            if report is not None:
                report.append(("flagged-row", it, done))
            return done
        assert kg == ko, f"iteration {it}: gpu committed {kg}, oracle {ko}"
        done += ko
    if div is None:
        assert gc[: len(ref.counts)] == list(ref.counts) or (tie_it is not None and len(gc) != len(ref.counts)), \
            "iteration counts differ"
    return div


def compare_with_resync(run_gpu, run_oracle, prompt, max_new: int, bf16: bool, max_flags: int, report=None):
    """Generation parity that continues past flagged near-ties.

    run_oracle(prompt, max_new, offset) -> GenResult of the oracle's decoding loop;
    run_gpu(prompt, max_new, offset) -> (tokens, per-iteration counts) of the device, both decoding
    `max_new` tokens after `prompt` with the same parameters (`offset` = new tokens already decided
    before `prompt` ends, for callers that index a truth continuation). Both runs are compared with
    compare_generation. At a flagged divergence both sides are re-synchronised on the oracle's prefix
    up to and including its decision at the near-tie (the device re-prefills that prefix), and the
    comparison continues from there until max_new tokens are decided. At most `max_flags` flagged
    positions are allowed; returns them as indexes into the new tokens."""
    prompt = [int(t) for t in prompt]
    done, flags = 0, []
    while done < max_new:
        ref = run_oracle(np.array(prompt, dtype=np.int32), max_new - done, done)
        tokens, counts = run_gpu(np.array(prompt, dtype=np.int32), max_new - done, done)
        div = compare_generation(tokens, counts, ref, bf16)
        if div is None:
            break
        flags.append(done + div)
        if report is not None:
            report.append(("flagged", done + div, ref.margins[div] if div < len(ref.margins) else None))
        assert len(flags) <= max_flags, f"more than {max_flags} flagged near-ties: {flags}"
        prompt += [int(t) for t in ref.tokens[: div + 1]]
        done += div + 1
    return flags
