"""Where a decode iteration's time goes, measured inside the replayed iteration graph.

Builds the timeline variant of libjf (JF_TIMELINE: thread 0 of every CTA records its entry time,
the time it got past its dependency wait and its exit time; see jf_tl_enable in include/jf.h),
decodes a few iterations of a random-weight model, and prints for each kernel of a layer the
median over layers of
  gap  = previous kernel's last CTA exit -> this kernel's first CTA past its dependency wait,
  work = that moment -> this kernel's last CTA exit,
plus the iteration's span. The instrumented library is separate from the default build; the
records cost a few atomics per CTA, so absolute times run slightly above the uninstrumented ones.

    python -m paper_2512_14681_gb300.timeline [--shape qwen2.5-7b-shape-bf16] [--prompt 1024] [--block 32]
"""
from __future__ import annotations

import argparse
import collections
import ctypes as C
import json
import sys

import numpy as np

MAX_RECORDS = 2000000  # JF_TL_MAX_RECORDS of include/jf.h
REC = np.dtype([("kid", "<u4"), ("blk", "<u4"), ("smid", "<u4"), ("pad", "<u4"),
                ("t0", "<u8"), ("t1", "<u8"), ("t2", "<u8")])
NAMES = {1: "rmsnorm", 2: "rmsnorm+partials", 3: "qkv finish", 5: "attention", 10: "gemm store", 11: "gemm resid",
         12: "gemm qkv", 13: "gate/up (swiglu)", 14: "lm head (argmax)", 15: "gemm partials", 20: "embedding",
         21: "acceptance", 22: "kv commit"}


def launches(rec):
    """Group records into launches: ordered by the time past the dependency wait, consecutive records
    of one kernel id belong to one launch (a launch passes its wait only after the previous one ended)."""
    r = rec[np.argsort(rec["t1"], kind="stable")]
    out = []
    for x in r:
        if not out or out[-1]["kid"] != int(x["kid"]):
            out.append({"kid": int(x["kid"]), "t1": int(x["t1"]), "t2": int(x["t2"]), "n": 0})
        L = out[-1]
        L["t2"] = max(L["t2"], int(x["t2"]))
        L["n"] += 1
    return out


def roles(seq):
    """Name each launch of one iteration by its place in the layer (the projections with split-K
    partials are told apart by the kernel before them)."""
    names, prev = [], None
    for L in seq:
        k = L["kid"]
        nm = NAMES.get(k, f"kernel {k}")
        if k == 15:
            nm = {2: "qkv", 1: "qkv", 5: "o proj"}.get(prev, "down")
        elif k == 2:
            nm = "norm2 (+o partials)" if prev == 15 and names and names[-1] == "o proj" else "norm1 (+down partials)"
        names.append(nm)
        prev = k
    return names


def summarize(rec):
    ls = launches(rec)
    ends = [i for i, L in enumerate(ls) if L["kid"] == 14]
    if len(ends) < 2:
        raise RuntimeError("fewer than two LM-head launches recorded")
    a, b = ends[-2], ends[-1]
    seq = ls[a + 1: b + 1]
    stats = collections.defaultdict(list)
    prev_end = ls[a]["t2"]
    for L, nm in zip(seq, roles(seq)):
        stats[nm].append(((L["t1"] - prev_end) / 1000.0, (L["t2"] - L["t1"]) / 1000.0))
        prev_end = L["t2"]
    table = {nm: {"count": len(v), "gap_us": float(np.median([g for g, _ in v])),
                  "work_us": float(np.median([w for _, w in v]))} for nm, v in stats.items()}
    return {"iteration_us": (ls[b]["t2"] - ls[a]["t2"]) / 1000.0, "launches": b - a, "kernels": table}


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--shape", default="qwen2.5-7b-shape-bf16")
    ap.add_argument("--prompt", type=int, default=1024)
    ap.add_argument("--block", type=int, default=32)
    ap.add_argument("--iters", type=int, default=4, help="decode iterations recorded (window mode)")
    args = ap.parse_args(argv)

    import torch

    from . import _lib
    from . import build as B
    from . import inputs as I

    _lib.LIB_PATH = B.build(timeline=True)
    from .jacobi import Context, Gen

    shape = I.SHAPES[args.shape]
    ctx = Context(shape, max_seqs=1, max_ctx=args.prompt + 512, max_rows=512)
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    prompt = I.prompt_tokens(shape.vocab, args.prompt, seed=100)
    L = _lib.load()
    ctx.generate([prompt], Gen(block_size=args.block, mode="window", max_new=2 * args.block))  # graphs, warm-up
    # the kernels write up to JF_TL_MAX_RECORDS records: the buffer holds all of them
    buf = torch.zeros(MAX_RECORDS * REC.itemsize, dtype=torch.uint8, device="cuda")
    cnt = torch.zeros(4, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    if L.jf_tl_enable(C.c_void_p(buf.data_ptr()), C.c_void_p(cnt.data_ptr())) != _lib.JF_OK:
        raise RuntimeError("jf_tl_enable failed (not a timeline build?)")
    try:
        out = ctx.generate([prompt], Gen(block_size=args.block, mode="window", max_new=args.iters))
        torch.cuda.synchronize()
    finally:
        L.jf_tl_enable(None, None)
    n = min(int(cnt[0].item()), MAX_RECORDS)
    rec = np.frombuffer(buf[: n * REC.itemsize].cpu().numpy().tobytes(), dtype=REC)
    res = summarize(rec)
    res["decode_ms_per_iteration_instrumented"] = out.decode_ms / max(out.iterations, 1)
    res["config"] = {"shape": args.shape, "prompt": args.prompt, "block": args.block, "records": int(n)}
    print(f"iteration {res['iteration_us']:.1f} us over {res['launches']} launches")
    print(f"{'kernel':24s} {'count':>5s} {'gap us':>8s} {'work us':>8s}")
    for nm, v in res["kernels"].items():
        print(f"{nm:24s} {v['count']:5d} {v['gap_us']:8.2f} {v['work_us']:8.2f}")
    print(json.dumps(res))
    ctx.close()
    return 0


if __name__ == "__main__":
    sys.exit(main())
