"""The binding's ctypes structures have the layout of include/jf.h's structs (no GPU): a C program
compiled against the header prints sizeof and every field's offsetof, which must equal ctypes'."""
import os
import shutil
import subprocess

import pytest

from paper_2512_14681_gb300 import _lib as J

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
STRUCTS = {
    "jf_model_config": J.ModelConfig,
    "jf_runtime_config": J.RuntimeConfig,
    "jf_block": J.Block,
    "jf_gen_params": J.GenParams,
    "jf_gen_stats": J.GenStats,
}


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_ctypes_structs_match_the_header(tmp_path):
    lines = ['#include <stddef.h>', '#include <stdio.h>', '#include "jf.h"', "int main(void) {"]
    for cname, py in STRUCTS.items():
        lines.append(f'  printf("{cname} sizeof %zu\\n", sizeof({cname}));')
        for f, _ in py._fields_:
            lines.append(f'  printf("{cname} {f} %zu\\n", offsetof({cname}, {f}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True,
                   capture_output=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    got = {}
    for ln in out:
        if ln.strip():
            s, f, v = ln.split()
            got[(s, f)] = int(v)
    for cname, py in STRUCTS.items():
        assert got[(cname, "sizeof")] == J.C.sizeof(py), cname
        for f, _ in py._fields_:
            assert got[(cname, f)] == getattr(py, f).offset, (cname, f)


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_oracle_config_struct_matches_its_c_definition(tmp_path):
    from oracle import oracle as O

    fields = [f for f, _ in O._Cfg._fields_]
    lines = ['#include <stddef.h>', '#include <stdio.h>', '#include "%s"' % os.path.join(ROOT, "oracle", "jf_oracle.c"),
             "int main(void) {", '  printf("sizeof %zu\\n", sizeof(orc_config));']
    lines += [f'  printf("{f} %zu\\n", offsetof(orc_config, {f}));' for f in fields]
    lines += ["  return 0;", "}"]
    src = tmp_path / "orc_layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "orc_layout"
    subprocess.run(["gcc", "-std=c11", str(src), "-o", str(exe), "-lm"], check=True, capture_output=True)
    got = dict(ln.split() for ln in subprocess.run([str(exe)], check=True, capture_output=True,
                                                   text=True).stdout.split("\n") if ln.strip())
    assert int(got["sizeof"]) == O.C.sizeof(O._Cfg)
    for f in fields:
        assert int(got[f]) == getattr(O._Cfg, f).offset, f
