"""Compile the decoding state machine of csrc/jf_decode.cu for the CPU (tests only).

The kernels there are written for one CTA per call; compiled as plain C++ with the host stand-in
of the device header (jf_device.cuh here) they run as a single thread, which visits every index
of their block-strided loops in order. The copy of the source differs from the file in three
places, each asserted below:
  * only the kernels are kept (the file is cut before the host launch helpers, which use the
    CUDA launch syntax);
  * the dynamic shared-memory arrays become pointers to a host buffer;
  * the draft-injection rule is renamed and reached through a hook, so a test can script the
    injected tokens (the rule itself stays callable and is checked on its own).
"""
import ctypes
import os
import re
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
CSRC = os.path.join(ROOT, "paper_2512_14681_gb300", "csrc")
OUT = os.path.join(HERE, "_build")
LIB = os.path.join(OUT, "libdecode_host.so")

_RULE = "__device__ int inject_token(const GenCfg& g, int seq, int x, int P0, int it, int* err) {"


def _cuda_include():
    for d in (os.environ.get("CUDA_HOME"), "/usr/local/cuda"):
        if d and os.path.exists(os.path.join(d, "include", "cuda_runtime.h")):
            return os.path.join(d, "include")
    raise RuntimeError("cuda_runtime.h not found (set CUDA_HOME)")


def prepare():
    os.makedirs(OUT, exist_ok=True)
    src = open(os.path.join(CSRC, "jf_decode.cu")).read()
    cut = src.index("cudaLaunchConfig_t pdl_cfg(")
    body = src[:cut] + "}  // namespace\n}  // namespace jf\n"
    body, n = re.subn(r"extern __shared__ int (\w+)\[\];", r"int* \1 = jf_host::dyn_smem();", body)
    assert n == 3, "dynamic shared-memory declarations changed"
    assert body.count(_RULE) == 1, "injection rule signature changed"
    body = body.replace(
        _RULE,
        "__device__ int inject_token_rule(const GenCfg& g, int seq, int x, int P0, int it, int* err);\n"
        "__device__ int inject_token(const GenCfg& g, int seq, int x, int P0, int it, int* err) {\n"
        "  return jf_host::scripted_inject(g, seq, x, P0, it, err, inject_token_rule);\n"
        "}\n"
        "__device__ int inject_token_rule(const GenCfg& g, int seq, int x, int P0, int it, int* err) {")
    assert "<<<" not in body
    open(os.path.join(OUT, "jf_decode_host.inc"), "w").write(body)
    for f in ("jf_decode.h", "jf_internal.h"):
        shutil.copy(os.path.join(CSRC, f), os.path.join(OUT, f))
    shutil.copy(os.path.join(HERE, "jf_device.cuh"), os.path.join(OUT, "jf_device.cuh"))


def build():
    prepare()
    cmd = ["g++", "-std=c++17", "-O1", "-shared", "-fPIC", "-Wno-attributes",
           "-include", os.path.join(HERE, "jf_host_pre.h"), "-I", OUT, "-I", _cuda_include(),
           os.path.join(HERE, "harness.cpp"), "-o", LIB]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    return LIB


def load():
    lib = ctypes.CDLL(build())
    P = ctypes.POINTER
    i32 = ctypes.c_int
    ip = P(ctypes.c_int)
    u64 = ctypes.c_ulonglong
    lib.hd_setup.argtypes = [i32] * 8 + [u64, u64] + [i32] * 4 + [ip, i32, i32, i32, i32]
    lib.hd_setup.restype = i32
    lib.hd_script.argtypes = [i32, ip, ip, ip]
    lib.hd_script.restype = None
    lib.hd_init.argtypes = [ip, ip, ip]
    lib.hd_init.restype = i32
    lib.hd_accept.argtypes = [ip, i32]
    lib.hd_accept.restype = i32
    lib.hd_view.argtypes = [ip] * 9
    lib.hd_view.restype = None
    lib.hd_out_tokens.argtypes = [ip]
    lib.hd_out_tokens.restype = None
    lib.hd_step.argtypes = [i32, ip, ip, i32, ip, ip, ip, ip, ip]
    lib.hd_step.restype = None
    lib.hd_inject_rule.argtypes = [u64, u64, i32, i32, i32, i32]
    lib.hd_inject_rule.restype = i32
    return lib
