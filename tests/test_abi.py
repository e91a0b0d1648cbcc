"""The C ABI library builds, loads and exports exactly what
include/layercheck.h declares, and the Python binding's structures match
the C layout.  No compute call is made (no GPU needed)."""
import ctypes as C
import os
import re
import subprocess
import tempfile

import pytest

from tests.conftest import ROOT

HEADER = os.path.join(ROOT, "include", "layercheck.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return set(re.findall(r"\b(lc_[a-z0-9_]+)\s*\(", text))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_27193_gb300 import build as B
    B.build()
    from paper_2609_27193_gb300 import _abi
    return _abi.load()


def test_header_declares_the_path(lib):
    names = declared_functions()
    for required in ("lc_register_layout", "lc_measure", "lc_select", "lc_pack_async",
                     "lc_pack_device", "lc_commit_snapshot", "lc_restore", "lc_wait_durable"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    names = declared_functions()
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    out = subprocess.run(["nm", "-D", "--defined-only", lib._name], capture_output=True,
                         text=True).stdout
    exported = {l.split()[-1] for l in out.splitlines() if l.strip()}
    assert exported == names, "exports differ from the header: %s" % (exported ^ names)


def test_binding_covers_the_header(lib):
    from paper_2609_27193_gb300 import _abi
    assert set(_abi.SIGNATURES) == declared_functions()


def test_struct_layout_matches_c(lib):
    from paper_2609_27193_gb300 import _abi
    structs = {"lc_segment": _abi.lc_segment, "lc_config": _abi.lc_config,
               "lc_select_info": _abi.lc_select_info, "lc_version": _abi.lc_version,
               "lc_counters": _abi.lc_counters, "lc_manifest_record": _abi.lc_manifest_record}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "layercheck.h"',
             "int main(void) {"]
    for name, cls in structs.items():
        lines.append('printf("%s %%zu\\n", sizeof(%s));' % (name, name))
        for f, _ in cls._fields_:
            lines.append('printf("%s.%s %%zu\\n", offsetof(%s, %s));' % (name, f, name, f))
    lines.append("return 0; }")
    with tempfile.TemporaryDirectory() as d:
        src = os.path.join(d, "layout.c")
        exe = os.path.join(d, "layout")
        open(src, "w").write("\n".join(lines))
        subprocess.run(["gcc", "-std=c11", "-I", os.path.dirname(HEADER), src, "-o", exe], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout
    got = dict(l.split() for l in out.splitlines())
    for name, cls in structs.items():
        assert int(got[name]) == C.sizeof(cls), name
        for f, _ in cls._fields_:
            assert int(got["%s.%s" % (name, f)]) == getattr(cls, f).offset, (name, f)


def test_header_compiles_as_c_and_cpp(lib):
    with tempfile.TemporaryDirectory() as d:
        src = os.path.join(d, "t.c")
        open(src, "w").write('#include "layercheck.h"\nint main(void){lc_config c; lc_config_default(&c);'
                             ' return c.pack_align == 256 ? 0 : 1;}\n')
        subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.dirname(HEADER), "-c",
                        src, "-o", os.path.join(d, "t.o")], check=True)
        subprocess.run(["g++", "-x", "c++", "-std=c++17", "-Wall", "-Werror", "-I",
                        os.path.dirname(HEADER), "-c", src, "-o", os.path.join(d, "t2.o")], check=True)


def test_defaults_and_errors_without_gpu(lib):
    from paper_2609_27193_gb300 import _abi
    cfg = _abi.lc_config()
    lib.lc_config_default(C.byref(cfg))
    assert cfg.eps_w == 1e-8 and cfg.pack_align == 256 and cfg.fuse_commit == 1
    assert cfg.mode == _abi.LC_DRIFT_SNAPSHOT and cfg.staging_bytes == 512 << 20
    ctx = C.c_void_p()
    assert lib.lc_create(None, 0, None, None) == _abi.LC_ERR_INVALID_ARG
    assert b"NULL" in lib.lc_last_error()
    bad = _abi.lc_config()
    lib.lc_config_default(C.byref(bad))
    bad.pack_align = 100
    assert lib.lc_create(C.byref(ctx), 0, None, C.byref(bad)) == _abi.LC_ERR_INVALID_ARG
    # NULL handles are rejected, not dereferenced
    assert lib.lc_measure(None, 1) == _abi.LC_ERR_INVALID_ARG
    assert lib.lc_select(None, 1e-3, 1, None, None, None) == _abi.LC_ERR_INVALID_ARG
    assert lib.lc_store_num_versions(None) == 0
    lib.lc_destroy(None)
    lib.lc_store_destroy(None)


def test_config_validation_without_gpu(lib):
    """lc_create checks its configuration before it touches a device."""
    from paper_2609_27193_gb300 import _abi
    cfg = _abi.lc_config()
    lib.lc_config_default(C.byref(cfg))
    assert cfg.copy_engine == _abi.LC_COPY_BULK and cfg.debug_flags == 0
    ctx = C.c_void_p()
    for field, value, word in (("copy_engine", 7, b"copy engine"), ("debug_flags", 8, b"debug flags"),
                               ("timeout_ms", 0, b"timeout_ms"), ("staging_bytes", 1 << 20, b"staging_bytes")):
        bad = _abi.lc_config()
        lib.lc_config_default(C.byref(bad))
        setattr(bad, field, value)
        assert lib.lc_create(C.byref(ctx), 0, None, C.byref(bad)) == _abi.LC_ERR_INVALID_ARG, field
        assert word in lib.lc_last_error(), (field, lib.lc_last_error())
    import paper_2609_27193_gb300 as P
    with pytest.raises(ValueError):
        P.LayerCheck(copy_engine="tma")


def test_product_path_has_no_fallback():
    """The package never imports the oracle, and fails loudly when the
    library is missing."""
    pkg = os.path.join(ROOT, "paper_2609_27193_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                text = open(os.path.join(dirpath, f)).read()
                assert "oracle" not in text.lower().replace("oracle-free", ""), f
    src = open(os.path.join(pkg, "_abi.py")).read()
    assert "raise ImportError" in src and "no CPU fallback" in src


def test_segment_validation_without_gpu():
    """The binding checks what a raw pointer cannot carry: moment dtypes and
    sizes, contiguity, one device, and both moments or neither; a segment
    keeps its tensors alive."""
    torch = pytest.importorskip("torch")
    import paper_2609_27193_gb300 as P
    w = torch.zeros(8, dtype=torch.bfloat16)
    r = torch.zeros(8, dtype=torch.bfloat16)
    m = torch.zeros(8, dtype=torch.float32)
    v = torch.zeros(8, dtype=torch.float32)
    s = P.segment(0, w, r, m, v)
    assert s.numel == 8 and s._refs[0] is w
    bad = [
        (w, r, m.to(torch.bfloat16), v),          # moments must be fp32
        (w, r, m, v[:4]),                         # and as long as w
        (w, r, m, None),                          # both or neither
        (w, r[:4], m, v),                         # snapshot as long as w
        (w, r.float(), m, v),                     # and of w's dtype
        (w, torch.zeros(16, dtype=torch.bfloat16)[::2], m, v),   # contiguous
    ]
    for args in bad:
        with pytest.raises(ValueError):
            P.segment(0, *args)
    with pytest.raises(TypeError):
        P.segment(0, w.to(torch.float16), None, m, v)
