"""The C ABI without a GPU: the library builds, loads and exports every function
include/lv.h declares, and the binding's struct layouts match the header's."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "lv.h")


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(lv_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    from paper_2606_22983_gb300 import build
    path = build()
    return ctypes.CDLL(path)


def test_every_declared_symbol_is_exported(lib):
    names = _declared_functions()
    assert len(names) >= 20
    for n in names:
        assert hasattr(lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", os.path.join(ROOT, "paper_2606_22983_gb300", "liblv.so")],
                         capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (lv_[a-z_]+)", out))
    assert set(names) <= exported


def test_binding_names_match_header():
    from paper_2606_22983_gb300 import lv
    assert sorted(lv.EXPORTED) == _declared_functions()
    for n in lv.EXPORTED:
        assert callable(getattr(lv, n)), n
    import re
    with open(HEADER) as f:
        m = re.search(r"#define LV_VERSION (\d+)", f.read())
    assert m and int(m.group(1)) == lv.LV_VERSION


def test_struct_layouts_match_header(tmp_path):
    from paper_2606_22983_gb300 import lv
    src = tmp_path / "layout.c"
    src.write_text(r'''
#include <stdio.h>
#include <stddef.h>
#include "lv.h"
#define F(T, m) printf(#T "." #m " %zu %zu\n", offsetof(T, m), sizeof(((T*)0)->m))
int main(void) {
  printf("sizeof lv_pool_desc %zu\n", sizeof(lv_pool_desc));
  printf("sizeof lv_session_state %zu\n", sizeof(lv_session_state));
  printf("sizeof lv_event %zu\n", sizeof(lv_event));
  printf("sizeof lv_victim %zu\n", sizeof(lv_victim));
  printf("sizeof lv_remap_entry %zu\n", sizeof(lv_remap_entry));
  printf("sizeof lv_stats %zu\n", sizeof(lv_stats));
  printf("sizeof lv_resident_result %zu\n", sizeof(lv_resident_result));
  printf("sizeof lv_request %zu\n", sizeof(lv_request));
  printf("sizeof lv_sched_params %zu\n", sizeof(lv_sched_params));
  F(lv_request, play_buffer_us); F(lv_request, kv_needed);
  F(lv_resident_result, k); F(lv_resident_result, n_found); F(lv_resident_result, n_victims);
  F(lv_resident_result, n_loaded); F(lv_resident_result, n_appended); F(lv_resident_result, status);
  F(lv_resident_result, sid);
  printf("sizeof lv_turn_desc %zu\n", sizeof(lv_turn_desc));
  printf("sizeof lv_controller_desc %zu\n", sizeof(lv_controller_desc));
  printf("sizeof lv_controller_counters %zu\n", sizeof(lv_controller_counters));
  printf("sizeof lv_controller_record %zu\n", sizeof(lv_controller_record));
  printf("sizeof lv_rank_params %zu\n", sizeof(lv_rank_params));
  F(lv_rank_params, num_sessions); F(lv_rank_params, flags); F(lv_rank_params, reply_prior_us);
  F(lv_rank_params, unit_us); F(lv_rank_params, policy); F(lv_rank_params, reserved);
  F(lv_controller_record, kind); F(lv_controller_record, sid); F(lv_controller_record, start_us);
  F(lv_controller_record, finish_us); F(lv_controller_record, deadline_us); F(lv_controller_record, n);
  F(lv_controller_record, data_offset);
  F(lv_turn_desc, sid); F(lv_turn_desc, num_candidates); F(lv_turn_desc, candidates);
  F(lv_turn_desc, now_us); F(lv_turn_desc, reply_audio_us); F(lv_turn_desc, reply_units);
  F(lv_turn_desc, append_tokens); F(lv_turn_desc, flags); F(lv_turn_desc, load_keys);
  F(lv_session_state, ctx_tokens); F(lv_session_state, flags); F(lv_session_state, gen_us);
  F(lv_session_state, play_us); F(lv_session_state, t_done_us); F(lv_session_state, reply_ema_us);
  F(lv_session_state, reply_n); F(lv_session_state, reply_tokens); F(lv_session_state, protect_until_us);
  F(lv_session_state, last_use_us);
  F(lv_event, kind); F(lv_event, sid); F(lv_event, t_us); F(lv_event, a); F(lv_event, b);
  F(lv_pool_desc, hbm_pages); F(lv_pool_desc, hbm_kv); F(lv_pool_desc, host_kv);
  F(lv_pool_desc, reply_prior_us); F(lv_pool_desc, t_play_mode); F(lv_pool_desc, policy);
  F(lv_pool_desc, tiers); F(lv_pool_desc, reserved);
  return 0;
}
''')
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.dirname(HEADER), str(src),
                    "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout
    got = {}
    for line in out.splitlines():
        parts = line.split()
        if parts[0] == "sizeof":
            got[parts[1]] = int(parts[2])
        else:
            got[parts[0]] = (int(parts[1]), int(parts[2]))
    assert got["lv_session_state"] == lv.SESSION_DTYPE.itemsize
    assert got["lv_event"] == lv.EVENT_DTYPE.itemsize
    assert got["lv_victim"] == lv.VICTIM_DTYPE.itemsize
    assert got["lv_remap_entry"] == lv.REMAP_DTYPE.itemsize
    assert got["lv_pool_desc"] == ctypes.sizeof(lv.lv_pool_desc)
    assert got["lv_stats"] == ctypes.sizeof(lv.lv_stats)
    assert got["lv_resident_result"] == lv.RESIDENT_DTYPE.itemsize
    assert got["lv_request"] == lv.REQUEST_DTYPE.itemsize == 48
    assert got["lv_sched_params"] == ctypes.sizeof(lv.lv_sched_params)
    assert got["lv_turn_desc"] == ctypes.sizeof(lv.lv_turn_desc)
    assert got["lv_controller_desc"] == ctypes.sizeof(lv.lv_controller_desc)
    assert got["lv_controller_counters"] == ctypes.sizeof(lv.lv_controller_counters)
    assert got["lv_controller_record"] == lv.CTL_RECORD_DTYPE.itemsize
    assert got["lv_rank_params"] == ctypes.sizeof(lv.lv_rank_params) == 48
    for name in ("num_sessions", "flags", "reply_prior_us", "unit_us", "policy", "reserved"):
        assert getattr(lv.lv_rank_params, name).offset == got[f"lv_rank_params.{name}"][0], name
    for name in lv.CTL_RECORD_DTYPE.names:
        assert lv.CTL_RECORD_DTYPE.fields[name][1] == got[f"lv_controller_record.{name}"][0], name
    for name, _ in lv.lv_turn_desc._fields_:
        assert getattr(lv.lv_turn_desc, name).offset == got[f"lv_turn_desc.{name}"][0], name
    assert got["lv_request.play_buffer_us"][0] == lv.REQUEST_DTYPE.fields["play_buffer_us"][1]
    assert got["lv_request.kv_needed"][0] == lv.REQUEST_DTYPE.fields["kv_needed"][1]
    for name in lv.RESIDENT_DTYPE.names:
        if name != "pad":
            assert lv.RESIDENT_DTYPE.fields[name][1] == got[f"lv_resident_result.{name}"][0], name
    for name in lv.SESSION_DTYPE.names:
        if name == "pad":
            continue
        off, size = got[f"lv_session_state.{name}"]
        assert lv.SESSION_DTYPE.fields[name][1] == off and lv.SESSION_DTYPE.fields[name][0].itemsize == size
    for name in lv.EVENT_DTYPE.names:
        off, size = got[f"lv_event.{name}"]
        assert lv.EVENT_DTYPE.fields[name][1] == off
    for name in ("hbm_pages", "hbm_kv", "host_kv", "reply_prior_us", "t_play_mode", "policy"):
        assert getattr(lv.lv_pool_desc, name).offset == got[f"lv_pool_desc.{name}"][0], name


def test_status_strings_and_argument_checks(lib):
    from paper_2606_22983_gb300 import lv
    for code, name in lv.STATUS_NAMES.items():
        assert lv.lv_status_str(code) == name
    assert lv.lv_version() == lv.LV_VERSION == 3
    # argument checks that need no device: a NULL descriptor / NULL out pointer
    L = lv.lib()
    h = ctypes.c_void_p()
    assert L.lv_pool_create(None, None, ctypes.byref(h)) == lv.LV_ERR_INVALID
    assert L.lv_pool_create(None, None, None) == lv.LV_ERR_INVALID
    assert L.lv_sync(None, None) == lv.LV_ERR_INVALID
    assert L.lv_remap(None, None, 0, None) == lv.LV_ERR_INVALID


def test_no_oracle_in_product_package():
    pkg = os.path.join(ROOT, "paper_2606_22983_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                text = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(from|import)\s+oracle\b", text, re.M), f
                assert "oracle/" not in text, f
