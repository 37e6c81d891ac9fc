"""Per-device one-time set-up (csrc/jf_once.h), compiled for the host and run without a GPU.

Kernel attributes (the tcgen05 GEMM's dynamic shared-memory limit) are set per device, so the
set-up guard of jf_op_gemm / jf_op_gemm_noalloc must remember each device on its own: a first call
on device 1 after device 0 must still run the set-up there, a failed set-up must run again, and
concurrent first calls on one device must run it once.
"""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2512_14681_gb300", "csrc")

PROGRAM = r"""
#include <atomic>
#include <cstdio>
#include <thread>
#include <vector>
#include "jf_once.h"

static std::atomic<int> calls[4];
static int fail_next = 0;

static int setup(int dev) {
  calls[dev]++;
  if (fail_next) { fail_next = 0; return 7; }
  return 0;
}

#define CHECK(c) do { if (!(c)) { std::printf("FAIL line %d: %s\n", __LINE__, #c); return 1; } } while (0)

int main() {
  jf::PerDeviceOnce once;
  // device 0, then device 1 with nothing else having run there: both set up, once each
  CHECK(once.run(0, [] { return setup(0); }) == 0);
  CHECK(once.run(0, [] { return setup(0); }) == 0);
  CHECK(calls[0] == 1);
  CHECK(once.run(1, [] { return setup(1); }) == 0);
  CHECK(calls[1] == 1);
  CHECK(once.run(1, [] { return setup(1); }) == 0);
  CHECK(calls[1] == 1);
  // a failed set-up is reported and not recorded: the next call retries
  fail_next = 1;
  CHECK(once.run(2, [] { return setup(2); }) == 7);
  CHECK(once.run(2, [] { return setup(2); }) == 0);
  CHECK(calls[2] == 2);
  CHECK(once.run(2, [] { return setup(2); }) == 0);
  CHECK(calls[2] == 2);
  // ordinals outside the table are refused without running the set-up
  CHECK(once.run(-1, [] { return setup(3); }) == -1);
  CHECK(once.run(jf::PerDeviceOnce::kMaxDevices, [] { return setup(3); }) == -1);
  CHECK(calls[3] == 0);
  // eight threads making their first call on one device: the set-up runs once
  std::vector<std::thread> ts;
  for (int t = 0; t < 8; ++t) ts.emplace_back([&] { once.run(3, [] { return setup(3); }); });
  for (auto& t : ts) t.join();
  CHECK(calls[3] == 1);
  std::printf("OK\n");
  return 0;
}
"""


def test_per_device_once(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no C++ compiler")
    src = tmp_path / "once.cpp"
    src.write_text(PROGRAM)
    exe = tmp_path / "once"
    subprocess.run([cxx, "-std=c++17", "-O1", "-pthread", "-I", CSRC, str(src), "-o", str(exe)], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0 and r.stdout.strip() == "OK", r.stdout + r.stderr
