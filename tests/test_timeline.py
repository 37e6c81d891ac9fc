"""The kernel-timeline tool (no GPU): the analysis of synthetic records, the ABI call in both builds."""
import ctypes as C

import numpy as np

from paper_2512_14681_gb300 import timeline as T


def _rec(kid, t1, t2, n=3, t0=None):
    r = np.zeros(n, dtype=T.REC)
    r["kid"], r["t0"], r["t1"], r["t2"] = kid, t1 - 100 if t0 is None else t0, t1, t2
    r["blk"] = np.arange(n)
    return r


def test_summary_of_a_synthetic_iteration():
    """Two iterations of a 1-layer forward; gaps and works come out of the second one."""
    seq = []
    t = 0
    def add(kid, gap, work):
        nonlocal t
        seq.append(_rec(kid, t + gap * 1000, t + (gap + work) * 1000))
        t += (gap + work) * 1000
    for _ in range(2):
        add(20, 1, 2)      # embedding
        add(1, 1, 4)       # norm1 (no partials: first layer)
        add(15, 1, 6)      # qkv
        add(3, 2, 2)       # finish
        add(5, 2, 10)      # attention
        add(15, 2, 6)      # o proj
        add(2, 1, 5)       # norm2
        add(13, 1, 44)     # gate/up
        add(15, 2, 22)     # down
        add(2, 2, 4)       # final norm
        add(14, 1, 180)    # lm head
        add(21, 1, 5)      # acceptance
        add(22, 1, 5)      # kv commit
    rec = np.concatenate(seq)
    rng = np.random.default_rng(0)
    rec = rec[rng.permutation(rec.size)]           # record order is arbitrary
    res = T.summarize(rec)
    k = res["kernels"]
    assert res["launches"] == 13
    assert k["qkv"]["work_us"] == 6 and k["o proj"]["gap_us"] == 2 and k["down"]["work_us"] == 22
    assert k["gate/up (swiglu)"]["work_us"] == 44 and k["attention"]["gap_us"] == 2
    assert k["norm2 (+o partials)"]["work_us"] == 5 and k["norm1 (+down partials)"]["count"] == 1
    assert k["lm head (argmax)"]["work_us"] == 180
    assert abs(res["iteration_us"] - sum(g + w for g, w in [(1, 2), (1, 4), (1, 6), (2, 2), (2, 10), (2, 6), (1, 5),
                                                            (1, 44), (2, 22), (2, 4), (1, 180)])
               - 12) < 1e-9  # + acceptance and commit of the previous iteration (1 + 5, 1 + 5)


def test_default_library_has_no_timeline():
    from paper_2512_14681_gb300 import _lib
    from paper_2512_14681_gb300 import build as B

    B.build()
    L = _lib.load()
    assert L.jf_tl_enable(None, None) == _lib.JF_EUNSUPPORTED


def test_timeline_build_exports_the_call():
    from paper_2512_14681_gb300 import build as B

    L = C.CDLL(B.build(timeline=True))
    L.jf_tl_enable.argtypes = [C.c_void_p, C.c_void_p]
    assert L.jf_tl_enable(C.c_void_p(16), None) == 1   # JF_EINVAL: one pointer without the other, host check
