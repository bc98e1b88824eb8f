"""The binding against the C header, without a GPU: every constant the binding repeats has the
header's value, and every struct the binding mirrors has the C compiler's size and field
offsets (a C program built from include/iq.h prints them)."""
import ctypes as C
import os
import re
import shutil
import subprocess

import pytest

from paper_2011_14504_gb300 import iq

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "iq.h")

STRUCTS = {"iq_conv_desc": iq.ConvDesc, "iq_bn_bits": iq.BnBits, "iq_term": iq.Term,
           "iq_kernel_time": iq.KernelTime}


def header_constants() -> dict:
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    vals = {}
    for body in re.findall(r"enum\s*\{(.*?)\}", src, flags=re.S):
        nxt = 0
        for item in body.split(","):
            item = item.strip()
            if not item:
                continue
            m = re.fullmatch(r"(IQ_\w+)\s*(?:=\s*(-?\d+))?", item)
            assert m, item
            v = int(m.group(2)) if m.group(2) is not None else nxt
            vals[m.group(1)] = v
            nxt = v + 1
    for name, v in re.findall(r"^#define\s+(IQ_\w+)\s+(-?\d+)\s*$", src, flags=re.M):
        vals[name] = int(v)
    return vals


def test_constants_match_the_header():
    vals = header_constants()
    assert len(vals) > 40
    shared = [n for n in vals if hasattr(iq, n)]
    assert {"IQ_OK", "IQ_ERR_CUDA", "IQ_MODE_RQ_GQ2", "IQ_BN_SCALES", "IQ_MAX_TERMS",
            "IQ_CONV_E_F16_READY", "IQ_KERNEL_CONV_SIMT"} <= set(shared)
    for n in shared:
        assert getattr(iq, n) == vals[n], n


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_struct_layouts_match_the_c_compiler(tmp_path):
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "iq.h"', "int main(void) {"]
    for cname, py in STRUCTS.items():
        lines.append(f'    printf("{cname} size %zu\\n", sizeof({cname}));')
        for fname, _ in py._fields_:
            lines.append(f'    printf("{cname} {fname} %zu\\n", offsetof({cname}, {fname}));')
    lines += ["    return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)],
                   check=True)
    got = {}
    for line in subprocess.run([str(exe)], check=True, capture_output=True,
                               text=True).stdout.splitlines():
        cname, field, v = line.split()
        got[(cname, field)] = int(v)
    for cname, py in STRUCTS.items():
        assert got[(cname, "size")] == C.sizeof(py), cname
        for fname, _ in py._fields_:
            assert got[(cname, fname)] == getattr(py, fname).offset, (cname, fname)
