"""The C-ABI library without a GPU: it builds for sm_103a, loads, exports
every entry point include/edp.h declares, its struct layouts match the
Python binding, and host-side argument validation answers synchronously."""
import ctypes as C
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "edp.h")


@pytest.fixture(scope="module")
def libpath():
    from paper_2609_24456_gb300 import build
    return build.build()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = set(re.findall(r"\b(edp_[a-z_]+)\s*\(", text))
    return sorted(n for n in names if not n.endswith("_fn"))


def test_every_declared_symbol_is_exported(libpath):
    names = declared_functions()
    assert len(names) >= 14
    out = subprocess.run(["nm", "-D", "--defined-only", libpath],
                         capture_output=True, text=True, check=True).stdout
    exported = set(line.split()[-1] for line in out.splitlines() if line.strip())
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    from paper_2609_24456_gb300 import edp
    assert set(edp.SIGNATURES) == set(names)
    L = C.CDLL(libpath)
    for n in names:
        assert getattr(L, n)


def test_struct_layouts_match_binding(tmp_path):
    from paper_2609_24456_gb300 import edp
    structs = {"edp_config": edp.edp_config, "edp_storage": edp.edp_storage,
               "edp_fields": edp.edp_fields, "edp_batch": edp.edp_batch,
               "edp_info": edp.edp_info, "edp_sched_costs": edp.edp_sched_costs,
               "edp_sched_choice": edp.edp_sched_choice,
               "edp_place_option": edp.edp_place_option,
               "edp_place_bw": edp.edp_place_bw, "edp_counters": edp.edp_counters}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "edp.h"',
             "int main(void) {"]
    for sname, cls in structs.items():
        lines.append('printf("%s %%zu\\n", sizeof(%s));' % (sname, sname))
        for fname, _ in cls._fields_:
            lines.append('printf("%s.%s %%zu\\n", offsetof(%s, %s));'
                         % (sname, fname, sname, fname))
    lines.append("return 0; }")
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe)], check=True)
    got = dict(l.rsplit(" ", 1) for l in
               subprocess.run([str(exe)], capture_output=True, text=True,
                              check=True).stdout.splitlines())
    for sname, cls in structs.items():
        assert int(got[sname]) == C.sizeof(cls), sname
        for fname, _ in cls._fields_:
            assert int(got["%s.%s" % (sname, fname)]) == getattr(cls, fname).offset, \
                (sname, fname)


def test_host_validation_without_gpu(libpath):
    from paper_2609_24456_gb300 import edp
    assert edp.edp_abi_version() == 2
    st = edp.edp_storage()
    bad = [
        edp.make_config(0, (1, 84, 84), edp.EDP_XFORM_STACK_F32),       # capacity 0
        edp.make_config(10, (3, 10, 10), edp.EDP_XFORM_CHW_NORM_BF16),  # 300 B
        edp.make_config(10, (1, 84, 84), edp.EDP_XFORM_STACK_F32,
                        frame_stack=17),
        edp.make_config(10, (3, 8, 8), edp.EDP_XFORM_HWC_CHW_BF16,
                        next_obs=True),
        edp.make_config(10, (1, 84, 84), edp.EDP_XFORM_STACK_F32,
                        hbm_capacity=11),
        edp.make_config(10, (5, 16, 16), edp.EDP_XFORM_CHW_NORM_BF16),  # c > 4
        edp.make_config(10, (3, 16, 16), edp.EDP_XFORM_CHW_NORM_BF16,
                        norm_std=(0.2, 0.0, 0.2)),
    ]
    for cfg in bad:
        out = C.c_void_p()
        s = edp.lib().edp_create(C.byref(cfg), C.byref(st), C.byref(out))
        assert s == edp.EDP_ERR_INVALID
        assert out.value is None
    cfg = edp.make_config(10, (1, 84, 84), edp.EDP_XFORM_STACK_F32)
    cfg.reserved[3] = 1
    out = C.c_void_p()
    assert edp.lib().edp_create(C.byref(cfg), C.byref(st), C.byref(out)) == \
        edp.EDP_ERR_INVALID
    # NULL contexts and arguments are refused, not dereferenced
    assert edp.lib().edp_sample(None, 0, 1, 0, 0, None, None, None) == edp.EDP_ERR_INVALID
    assert edp.lib().edp_sync(None, None) == edp.EDP_ERR_INVALID
    assert edp.lib().edp_destroy(None) == edp.EDP_ERR_INVALID
    assert edp.lib().edp_probe_host_read(None, 16, None, None) == edp.EDP_ERR_INVALID


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    from paper_2609_24456_gb300 import edp
    monkeypatch.setattr(edp, "_lib", None)
    monkeypatch.setattr(edp, "LIB_PATH", str(tmp_path / "nope.so"))
    with pytest.raises(RuntimeError):
        edp.lib()
