"""Strength of the oracle's transformer pins (no GPU): each plausible mistake below is planted into a
copy of oracle/jf_oracle.c, compiled on the CPU, and the pins of tests/test_oracle_pins.py and
tests/test_oracle_bias_tied.py must fail on it. A mistake that no pin notices would mean a hole in
the oracle's checks. A mistake is one (anchor, replacement) pair, or a list of them."""
import inspect
import os
import shutil
import subprocess

import pytest

from oracle import build as OB
from oracle import oracle as O

pytestmark = pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")

PLANTED = {
    "RMSNorm without eps": ("double r = 1.0 / sqrt(ss / d + eps);", "double r = 1.0 / sqrt(ss / d);"),
    "RMSNorm over the sum instead of the mean": ("double r = 1.0 / sqrt(ss / d + eps);",
                                                  "double r = 1.0 / sqrt(ss + eps);"),
    "RoPE on adjacent pairs": ("double x1 = v[i], x2 = v[i + h];\n        v[i] = x1 * c - x2 * s;\n"
                               "        v[i + h] = x2 * c + x1 * s;",
                               "double x1 = v[2 * i], x2 = v[2 * i + 1];\n        v[2 * i] = x1 * c - x2 * s;\n"
                               "        v[2 * i + 1] = x2 * c + x1 * s;"),
    "RoPE rotating the other way": ("v[i] = x1 * c - x2 * s;\n        v[i + h] = x2 * c + x1 * s;",
                                    "v[i] = x1 * c + x2 * s;\n        v[i + h] = x2 * c - x1 * s;"),
    "RoPE frequency exponent halved": ("double inv = pow(theta, -(2.0 * i) / (double)hd);",
                                       "double inv = pow(theta, -(1.0 * i) / (double)hd);"),
    "GQA head mapping interleaved": ("int kvh = h / group;", "int kvh = h % Hkv;"),
    "attention scores unscaled": ("double scale = 1.0 / sqrt((double)hd);", "double scale = 1.0;"),
    "causal mask excludes the row itself": ("int same = (seg[j] == seg[i]) && (pos[j] <= pos[i]);",
                                            "int same = (seg[j] == seg[i]) && (pos[j] < pos[i]);"),
    "ancestor segments invisible": ("int ancestor = (seg[j] != seg[i]) && ((anc[seg[i]] >> seg[j]) & 1u);",
                                    "int ancestor = 0;"),
    "attention residual dropped": ("orc_linear_t(M, att, orc_layer_t(m, l, L_WO), tmp);\n"
                                   "        for (long j = 0; j < (long)M * d; j++) x[j] += tmp[j];",
                                   "orc_linear_t(M, att, orc_layer_t(m, l, L_WO), tmp);\n"
                                   "        for (long j = 0; j < (long)M * d; j++) x[j] = tmp[j];"),
    "SiLU on the up projection instead of the gate": ("gt[j] = RB(orc_silu(gt[j]) * ut[j]);",
                                                      "gt[j] = RB(gt[j] * orc_silu(ut[j]));"),
    "argmax ties to the highest id": ("if (x > b1) { b2 = b1; b1 = x; best = v; }",
                                      "if (x >= b1) { b2 = b1; b1 = x; best = v; }"),
    "projection weights transposed": ("for (long k = 0; k < K; k++) wrow[k] = orc_w(W, n * K + k);",
                                      "for (long k = 0; k < K; k++) wrow[k] = orc_w(W, k * N + n);"),
    "values read from the keys": ("const double* vj = vptr[j] + (long)kvh * hd;",
                                  "const double* vj = kptr[j] + (long)kvh * hd;"),
    "MLP residual dropped": ("orc_linear_t(M, gt, orc_layer_t(m, l, L_WD), tmp);\n"
                             "        for (long j = 0; j < (long)M * d; j++) x[j] += tmp[j];",
                             "orc_linear_t(M, gt, orc_layer_t(m, l, L_WD), tmp);\n"
                             "        for (long j = 0; j < (long)M * d; j++) x[j] = tmp[j];"),
    "embedding row index": ("x[(long)i * d + j] = orc_w(&m->t[T_EMBED], (long)tokens[i] * d + j);",
                            "x[(long)i * d + j] = orc_w(&m->t[T_EMBED], (long)tokens[i] + j);"),
    "final-norm output not rounded to bf16": (
        "        for (int j = 0; j < d; j++) h[(long)i * d + j] = RB(h[(long)i * d + j]);\n    }\n    free(gt);",
        "    }\n    free(gt);"),
    "keys not rounded to bf16": ("kk[(long)i * kvd + j] = RB(kk[(long)i * kvd + j]);",
                                 "kk[(long)i * kvd + j] = kk[(long)i * kvd + j];"),
    "attention output not rounded to bf16": ("for (long j = 0; j < (long)M * qd; j++) att[j] = RB(att[j]);",
                                             "for (long j = 0; j < (long)M * qd; j++) att[j] = att[j];"),
    "SwiGLU product not rounded to bf16": ("gt[j] = RB(orc_silu(gt[j]) * ut[j]);", "gt[j] = orc_silu(gt[j]) * ut[j];"),
    "final norm skipped": ("orc_rmsnorm(d, x + (long)i * d, gain, cf->rms_eps, h + (long)i * d);\n"
                           "        for (int j = 0; j < d; j++) h[(long)i * d + j] = RB(h[(long)i * d + j]);\n"
                           "    }\n    free(gt);",
                           "for (int j = 0; j < d; j++) h[(long)i * d + j] = RB(x[(long)i * d + j]);\n"
                           "    }\n    free(gt);"),
    "query bias dropped": ("for (int j = 0; j < qd; j++) q[(long)i * qd + j] += orc_w(bq, j);", "(void)bq;"),
    "key bias dropped": ("kk[(long)i * kvd + j] += orc_w(bk, j);", "(void)bk;"),
    "value bias dropped": ("vv[(long)i * kvd + j] += orc_w(bv, j);", "(void)bv;"),
    "query and key biases added after the rotary embedding": [
        ("if (cf->qkv_bias) {\n            /* per-feature biases", "if (0) {\n            /* per-feature biases"),
        ("            for (int j = 0; j < qd; j++) q[(long)i * qd + j] = RB(q[(long)i * qd + j]);",
         "            if (cf->qkv_bias) {\n"
         "                for (int j = 0; j < qd; j++) q[(long)i * qd + j] += orc_w(orc_layer_t(m, l, L_BQ), j);\n"
         "                for (int j = 0; j < kvd; j++) kk[(long)i * kvd + j] += orc_w(orc_layer_t(m, l, L_BK), j);\n"
         "                for (int j = 0; j < kvd; j++) vv[(long)i * kvd + j] += orc_w(orc_layer_t(m, l, L_BV), j);\n"
         "            }\n"
         "            for (int j = 0; j < qd; j++) q[(long)i * qd + j] = RB(q[(long)i * qd + j]);")],
}


def _pins():
    import tests.test_oracle_bias_tied as B
    import tests.test_oracle_pins as T

    return [(f"{mod.__name__}.{n}", f) for mod in (T, B) for n, f in inspect.getmembers(mod, inspect.isfunction)
            if n.startswith("test_") and not inspect.signature(f).parameters]


@pytest.mark.parametrize("name", sorted(PLANTED))
def test_planted_mistake_fails_a_pin(name, tmp_path, monkeypatch):
    edits = PLANTED[name]
    src = open(OB.SRC).read()
    for a, b in ([edits] if isinstance(edits, tuple) else edits):
        assert src.count(a) == 1, "anchor of the planted mistake not found once"
        src = src.replace(a, b)
    c_path = tmp_path / "jf_oracle_planted.c"
    c_path.write_text(src)
    so = str(tmp_path / "libjforacle_planted.so")
    subprocess.run(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-ffp-contract=off", "-o", so,
                    str(c_path), "-lm"], check=True, capture_output=True)
    monkeypatch.setattr(OB, "build", lambda force=False: so)
    monkeypatch.setattr(O, "_lib", None)
    failed = []
    for n, f in _pins():
        try:
            f()
        except Exception:  # noqa: BLE001 - any failure of a pin counts as detection
            failed.append(n)
    assert failed, f"no pin notices: {name}"
