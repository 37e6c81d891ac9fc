"""Writes tests/golden/logit_noise_floor.json: how far the oracle's own fp32 logits move when each
value reaching a bf16 rounding point is perturbed by one fp32 unit (relative 2^-24), for the
forwards the wide parity tests check. Calls only oracle/ and the seeded inputs.

The paper fixes no precision. Under the bf16 reading (weights, KV cache and the activations that
enter a matrix product are bf16), an implementation that accumulates in fp32 reaches every rounding
point a few fp32 units away from the fp64 oracle, and a rounding that falls on the other side of a
bf16 boundary spreads through the next layers, more so the wider they are. The spread measured here
is therefore the distance any fp32 implementation can be expected to keep from the oracle; the wide
tests allow twice it where it exceeds the fixed 3e-2 bound.

    python tests/golden/logit_noise_floor.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import oracle as O  # noqa: E402
from paper_2512_14681_gb300 import inputs as I  # noqa: E402

EPS = 2.0 ** -24
SEEDS = (1, 2)

# (name, shape, cached tokens, prompt seed, rows, rows seed, prefill chunk): the forwards of
# tests/test_gpu_wide.py (7B widths, 1,100-token cache) and tests/test_gpu_large.py (full depth)
CASES = [
    ("wide-7b-2layer-32rows", I.QWEN7B_2L_BF16, 1100, 51, 32, 52, 384),
    ("full-1.5b-32rows", I.QWEN15B_BF16, 20, 33, 32, 34, 32),
    ("full-7b-32rows", I.QWEN7B_BF16, 20, 33, 32, 34, 32),
]


def logits(model, P, pseed, R, rseed, chunk, q0_first):
    shape_vocab = model.cfg.vocab
    prompt = I.prompt_tokens(shape_vocab, P, seed=pseed)
    oc = O.Cache(model, P + R + 8, max(chunk, R))
    last = None
    for s in range(0, P, chunk):
        e = min(P, s + chunk)
        last = O.forward(model, oc, prompt[s:e], np.arange(s, e))
        oc.commit(np.arange(e - s))
    rows = I.prompt_tokens(shape_vocab, R, seed=rseed)
    if q0_first:
        rows = np.concatenate([[int(last.argmax[-1])], I.prompt_tokens(shape_vocab, R - 1, seed=rseed)]).astype(np.int32)
    return O.forward(model, oc, rows, np.arange(P, P + R), want_logits=True).logits


def main():
    out = {"eps": EPS, "seeds": list(SEEDS), "cases": {}}
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "logit_noise_floor.json")
    if os.path.exists(path):
        out = json.load(open(path))
    only = set(sys.argv[1:])
    for name, shape, P, pseed, R, rseed, chunk in CASES:
        if only and name not in only:
            continue
        model = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)
        q0_first = name.startswith("wide")
        O.set_perturbation(0.0)
        ref = logits(model, P, pseed, R, rseed, chunk, q0_first)
        mx, sd = [], []
        for seed in SEEDS:
            O.set_perturbation(EPS, seed)
            d = np.abs(logits(model, P, pseed, R, rseed, chunk, q0_first) - ref)
            mx.append(float(d.max()))
            sd.append(float(d.std()))
        O.set_perturbation(0.0)
        out["cases"][name] = {"max_abs": max(mx), "std": max(sd), "per_seed_max": mx, "per_seed_std": sd}
        print(name, out["cases"][name], flush=True)
        del model
        json.dump(out, open(path, "w"), indent=1)


if __name__ == "__main__":
    main()
