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


def need_gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch


def compare_generation(gpu_tokens, gpu_counts, ref, bf16: bool, report=None):
    """Token sequences must match exactly up to the first divergence, which must sit at a
    flagged near-tie of the oracle; per-iteration counts must match for every iteration that
    ends before it. Returns the flagged position or None."""
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
    for it, (kg, ko) in enumerate(zip(gc, ref.counts)):
        if div is not None and done + ko >= div:
            break
        assert kg == ko, f"iteration {it}: gpu committed {kg}, oracle {ko}"
        done += ko
    if div is None:
        assert gc[: len(ref.counts)] == list(ref.counts)
    return div
