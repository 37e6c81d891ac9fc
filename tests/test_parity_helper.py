"""The GPU parity tests' comparison rule (tests/parity.py), on synthetic generations (no GPU):
tokens equal up to the first divergence, which must sit at one of the oracle's near-ties; committed
counts equal for every iteration that ends before it."""
import types

import pytest

from tests.parity import compare_generation, flag_tol


def ref(tokens, counts, margins):
    return types.SimpleNamespace(tokens=list(tokens), counts=list(counts), margins=list(margins))


def test_identical_generation_passes():
    r = ref([5, 6, 7, 8, 9], [2, 2, 1], [1.0] * 5)
    assert compare_generation([5, 6, 7, 8, 9], [2, 2, 1], r, bf16=True) is None


def test_divergence_at_a_near_tie_is_flagged_and_later_counts_are_free():
    tol = flag_tol(True)
    r = ref([5, 6, 7, 8, 9, 10], [2, 3, 1], [1.0, 1.0, 1.0, 1.0, tol / 2, 1.0])
    rep = []
    # token 4 differs at a near-tie; iteration 1 (tokens 2..4) may then commit a different count
    assert compare_generation([5, 6, 7, 8, 3, 3], [2, 1, 9], r, bf16=True, report=rep) == 4
    assert rep == [("flagged", 4, tol / 2)]


def test_divergence_at_a_clear_decision_fails():
    r = ref([5, 6, 7, 8], [2, 2], [1.0, 1.0, 1.0, 1.0])
    with pytest.raises(AssertionError):
        compare_generation([5, 6, 0, 8], [2, 2], r, bf16=False)


def test_fp32_tolerance_is_tighter_than_bf16():
    r = ref([5, 6, 7], [3], [1.0, 1e-3, 1.0])
    assert compare_generation([5, 0, 7], [3], r, bf16=True) == 1        # 1e-3 < 2 * 3e-2
    with pytest.raises(AssertionError):
        compare_generation([5, 0, 7], [3], r, bf16=False)              # 1e-3 > 2 * 1e-4


def test_count_mismatch_before_the_divergence_fails():
    r = ref([5, 6, 7, 8, 9], [1, 2, 2], [1.0, 1.0, 1.0, 1.0, 1e-9])
    with pytest.raises(AssertionError):
        compare_generation([5, 6, 7, 8, 0], [2, 1, 2], r, bf16=True)   # iteration 0 ends before token 4


def test_length_and_count_mismatch_without_divergence_fail():
    r = ref([5, 6, 7], [2, 1], [1.0] * 3)
    with pytest.raises(AssertionError):
        compare_generation([5, 6], [2, 1], r, bf16=True)
    with pytest.raises(AssertionError):
        compare_generation([5, 6, 7], [1, 2], r, bf16=True)


# ---- re-synchronisation after flagged near-ties (compare_with_resync) ----------------------------
from tests.parity import compare_with_resync  # noqa: E402


def _runners(truth, margins, gpu_flip, count=2):
    """Oracle: the truth continuation, `count` tokens per iteration. Device: the same, except that at
    the absolute new-token indexes in gpu_flip it decides another token (and keeps its own branch)."""
    calls = []

    def oracle(prompt, max_new, offset):
        toks = truth[offset: offset + max_new]
        cnt = [count] * (len(toks) // count) + ([len(toks) % count] if len(toks) % count else [])
        return ref(toks, cnt, margins[offset: offset + max_new])

    def gpu(prompt, max_new, offset):
        calls.append((len(prompt), max_new, offset))
        toks = list(truth[offset: offset + max_new])
        for i in gpu_flip:
            if offset <= i < offset + max_new:
                toks[i - offset:] = [t + 1000 for t in toks[i - offset:]]  # diverged branch
                break
        cnt = [count] * (len(toks) // count) + ([len(toks) % count] if len(toks) % count else [])
        return toks, cnt

    return oracle, gpu, calls


def test_resync_continues_after_each_flagged_tie():
    tol = flag_tol(True)
    truth = list(range(10, 30))
    margins = [1.0] * 20
    margins[3] = margins[11] = tol / 4
    oracle, gpu, calls = _runners(truth, margins, gpu_flip=[3, 11])
    rep = []
    flags = compare_with_resync(gpu, oracle, [1, 2, 3], 20, bf16=True, max_flags=2, report=rep)
    assert flags == [3, 11]
    # three runs: the whole generation, then from token 4 (prompt + 4 oracle tokens), then from 12
    assert calls == [(3, 20, 0), (7, 16, 4), (15, 8, 12)]
    assert [r[1] for r in rep] == [3, 11]


def test_resync_still_fails_a_clear_divergence_after_a_tie():
    tol = flag_tol(True)
    truth = list(range(10, 30))
    margins = [1.0] * 20
    margins[3] = tol / 4
    oracle, gpu, _ = _runners(truth, margins, gpu_flip=[3, 9])   # token 9 has a clear margin
    with pytest.raises(AssertionError):
        compare_with_resync(gpu, oracle, [1, 2, 3], 20, bf16=True, max_flags=4)


def test_resync_bounds_the_number_of_flags():
    tol = flag_tol(True)
    truth = list(range(10, 30))
    margins = [tol / 4] * 20
    oracle, gpu, _ = _runners(truth, margins, gpu_flip=[2, 5, 8])
    with pytest.raises(AssertionError):
        compare_with_resync(gpu, oracle, [1], 20, bf16=True, max_flags=2)
    assert compare_with_resync(gpu, oracle, [1], 20, bf16=True, max_flags=3) == [2, 5, 8]


def _with_rows(r, row_margins):
    """Attach per-iteration forward rows (only their margins matter to the rule) to a reference."""
    r.iters = [types.SimpleNamespace(rows={"margin": m}) for m in row_margins]
    return r


def test_count_mismatch_after_a_row_tie_is_flagged():
    tol = flag_tol(True)
    # same tokens; iteration 2 commits a different count; iteration 1 had a draft row at a near-tie
    r = _with_rows(ref([5, 6, 7, 8, 9, 10], [2, 1, 3], [1.0] * 6), [[1.0, 1.0], [1.0, tol / 3], [1.0, 1.0]])
    rep = []
    assert compare_generation([5, 6, 7, 8, 9, 10], [2, 1, 1, 2], r, bf16=True, report=rep) == 3
    assert rep == [("flagged-row", 2, 3)]


def test_count_mismatch_before_any_row_tie_fails():
    tol = flag_tol(True)
    r = _with_rows(ref([5, 6, 7, 8, 9, 10], [2, 1, 3], [1.0] * 6), [[1.0], [1.0], [tol / 3]])
    with pytest.raises(AssertionError):
        compare_generation([5, 6, 7, 8, 9, 10], [1, 2, 3], r, bf16=True)   # iteration 0 differs
