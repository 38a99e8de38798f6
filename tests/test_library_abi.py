"""CPU-side checks of the C ABI: the library builds, loads, exports every function that
include/*.h declares, and its structs have the layout the binding assumes.  No GPU."""
import glob
import ctypes
import os
import re
import subprocess

import pytest

from conftest import ROOT

HEADERS = sorted(glob.glob(os.path.join(ROOT, "include", "*.h")))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_37007_gb300 import build, mcd
    build.build()
    return mcd.load_library()


def declared_functions():
    names = set()
    for h in HEADERS:
        text = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names |= set(re.findall(r"\b(mcd_[a-z_0-9]+)\s*\(", text))
    return sorted(names)


def test_header_declares_the_boundary():
    fns = declared_functions()
    for need in ("mcd_create", "mcd_load_weights", "mcd_draft", "mcd_verify_accept", "mcd_decode_frame",
                 "mcd_accept_from_logits", "mcd_destroy", "mcd_status_str", "mcd_outer_create",
                 "mcd_outer_prefill", "mcd_pipeline_frames"):
        assert need in fns


def test_every_declared_symbol_is_exported(lib):
    missing = [f for f in declared_functions() if not hasattr(lib, f)]
    assert not missing, missing


def test_every_declared_symbol_has_a_binding_of_the_same_name():
    from paper_2609_37007_gb300 import mcd
    missing = [f for f in declared_functions() if not callable(getattr(mcd, f, None))]
    assert not missing, missing


def test_struct_layouts_match_the_binding(tmp_path):
    from paper_2609_37007_gb300 import mcd
    src = tmp_path / "sz.c"
    src.write_text('#include "mcd_pipeline.h"\n#include <stdio.h>\n#include <stddef.h>\n'
                   'int main(void){printf("%zu %zu %zu %zu %zu %zu",'
                   ' sizeof(mcd_config), sizeof(mcd_call_trace), sizeof(mcd_frame_stats),'
                   ' offsetof(mcd_config, seed), sizeof(mcd_outer_config), offsetof(mcd_outer_config, seed));'
                   'return 0;}\n')
    exe = tmp_path / "sz"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()
    cfg_sz, trace_sz, stats_sz, seed_off, ocfg_sz, oseed_off = map(int, out)
    assert ocfg_sz == ctypes.sizeof(mcd.McdOuterConfig)
    assert oseed_off == mcd.McdOuterConfig.seed.offset
    assert cfg_sz == ctypes.sizeof(mcd.McdConfig)
    assert seed_off == mcd.McdConfig.seed.offset
    assert trace_sz == mcd.CALL_TRACE_DTYPE.itemsize
    assert stats_sz == 32


def test_status_strings(lib):
    from paper_2609_37007_gb300 import mcd
    assert mcd.mcd_status_str(0) == "ok"
    assert "timed out" in mcd.mcd_status_str(5)
    assert mcd.mcd_status_str(99) == "unknown status"


def test_create_rejects_bad_configs_before_touching_a_device(lib):
    from paper_2609_37007_gb300 import mcd
    from paper_2609_37007_gb300.synth import MCD
    out = ctypes.c_void_p()
    for bad, want in ((MCD.replace(head_dim=96), 7), (MCD.replace(n_q_heads=15), 1),
                      (MCD.replace(draft_len=8), 7), (MCD.replace(top_k=300), 7),
                      (MCD.replace(temperature=0.0), 1), (MCD.replace(n_pos=16), 7)):
        c = mcd.config_struct(bad)
        assert lib.mcd_create(ctypes.byref(c), None, ctypes.byref(out)) == want
        assert not out.value
    assert lib.mcd_create(None, None, ctypes.byref(out)) == 1


def test_missing_library_fails_loudly(monkeypatch):
    from paper_2609_37007_gb300 import mcd
    monkeypatch.setattr(mcd, "_lib", None)
    monkeypatch.setattr(mcd, "_LIB_PATH", os.path.join(ROOT, "nonexistent", "libmcd.so"))
    with pytest.raises(RuntimeError, match="missing"):
        mcd.load_library()


def test_null_context_calls_return_errors(lib):
    assert lib.mcd_sync(None) == 1
    assert lib.mcd_decode_frame(None, 0, 0, None, None, None, None, None) == 1
    assert lib.mcd_num_ctas(None) == 0
    lib.mcd_destroy(None)
