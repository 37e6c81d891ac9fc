"""The attention's launch-form rule (csrc/jf_attn_form.h), compiled for the host and run without a GPU.

A unit (chain, KV head, 128-row query tile) runs on 8 CTAs; as an 8-CTA cluster only 15 fit on a
GB300's 152 SMs at once (cudaOccupancyMaxActiveClusters, measured), as independent CTAs all 152 do.
The rule takes the clustered form unless the unclustered one needs fewer waves of units. The cases
below are the 7B shape (4 KV heads, 7 query heads each) at the sweep's measured points, where the
form it picks was the faster one, and the small model's 256-row window that the GPU test of the
unclustered form relies on.
"""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2512_14681_gb300", "csrc")

PROGRAM = r"""
#include <cstdio>
#include "jf_attn_form.h"

#define CHECK(c) do { if (!(c)) { std::printf("FAIL line %d: %s\n", __LINE__, #c); return 1; } } while (0)

static bool clustered(int M, int chains, int Hkv, int G) {
  const int bound = Hkv * ((M * G + 127) / 128 + chains);
  const int units = jf::attn_units_estimate(M, chains, bound, Hkv, G, 128);
  return jf::attn_use_clusters(units, 8, 15, 152);
}

int main() {
  // unit estimates: rows spread over the chains, whole 128-row tiles per chain and KV head
  CHECK(jf::attn_units_estimate(32, 1, 12, 4, 7, 128) == 8);      // 224 query rows: 2 tiles x 4 heads
  CHECK(jf::attn_units_estimate(64, 4, 32, 4, 7, 128) == 16);     // 4 windows of 16 rows: 1 tile each
  CHECK(jf::attn_units_estimate(128, 4, 44, 4, 7, 128) == 32);    // 4 windows of 32 rows: 2 tiles each
  CHECK(jf::attn_units_estimate(512, 4, 132, 4, 7, 128) == 112);  // 4 windows of 128 rows: 7 tiles each
  CHECK(jf::attn_units_estimate(512, 4, 100, 4, 7, 128) == 100);  // capped by the launch bound
  CHECK(jf::attn_units_estimate(5, 0, 8, 2, 4, 128) == 2);        // no chain count: one chain
  // waves: clustered ceil(u / 15), unclustered ceil(8 u / 152); ties to the clustered form
  CHECK(jf::attn_use_clusters(15, 8, 15, 152));                    // 1 wave either way
  CHECK(!jf::attn_use_clusters(16, 8, 15, 152));                   // 2 waves against 1
  CHECK(jf::attn_use_clusters(28, 8, 15, 152));                    // 2 against 2
  CHECK(!jf::attn_use_clusters(112, 8, 15, 152));                  // 8 against 6
  CHECK(jf::attn_use_clusters(3, 8, 0, 152) == jf::attn_use_clusters(3, 8, 1, 152));  // no count: 1
  // the sweep's points (7B shape): the form the rule picks is the one measured faster
  CHECK(clustered(32, 1, 4, 7));      // decode, 32 rows
  CHECK(!clustered(64, 1, 4, 7));     // 64-row window: 3.96 (clustered) against 3.73 ms
  CHECK(clustered(128, 1, 4, 7));     // 128-row window: the clustered fold 5% faster at equal waves
  CHECK(clustered(192, 1, 4, 7));     // 192 rows: 5.55 against 5.70 ms
  CHECK(!clustered(64, 4, 4, 7));     // B = 4, n = 16: at 32k 8.83 against 6.07 ms
  CHECK(!clustered(128, 4, 4, 7));    // B = 4, n = 32
  CHECK(!clustered(512, 4, 4, 7));    // B = 4, n = 128: at 32k 29.21 against 24.44 ms
  CHECK(!clustered(384, 1, 4, 7));    // the knee's 384 rows: 9.75 against 9.20 ms
  // the small model (2 KV heads, 4 query heads each): a 256-row window is unclustered, one row is not
  CHECK(!clustered(256, 1, 2, 4));
  CHECK(clustered(1, 1, 2, 4));
  std::printf("ok\n");
  return 0;
}
"""


@pytest.mark.skipif(shutil.which("g++") is None, reason="needs g++")
def test_attention_form_rule(tmp_path):
    src = tmp_path / "form.cpp"
    src.write_text(PROGRAM)
    exe = tmp_path / "form"
    subprocess.run(["g++", "-std=c++17", "-O1", "-I", CSRC, str(src), "-o", str(exe)], check=True,
                   capture_output=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0 and out.stdout.strip() == "ok", out.stdout
