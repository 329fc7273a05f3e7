"""The C ABI library loads and exports every symbol include/adept.h declares; host-side
argument checks that need no GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2601_03700_gb300 import build
    build.build()
    import paper_2601_03700_gb300 as adept
    return adept.load_library()


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "adept.h")).read()
    return sorted(set(re.findall(r"ADEPT_API\s+[\w\s\*]+?\b(adept_\w+)\s*\(", src)))


def test_header_declares_the_five_calls():
    names = declared_symbols()
    for n in ("adept_model_load", "adept_prefill", "adept_decode_step", "adept_skip_kv_fill", "adept_free"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    import paper_2601_03700_gb300 as adept
    names = declared_symbols()
    assert len(names) >= 14
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(adept.ABI_SYMBOLS) == names


def test_option_numbers_match_the_header():
    """Every ADEPT_OPT_* of include/adept.h has the same number as the binding's OPT_*."""
    import paper_2601_03700_gb300 as adept
    src = open(os.path.join(ROOT, "include", "adept.h")).read()
    opts = dict(re.findall(r"ADEPT_OPT_(\w+)\s*=\s*(\d+)", src))
    assert len(opts) >= 13
    for name, val in opts.items():
        assert getattr(adept, "OPT_" + name) == int(val), name


def test_status_strings_and_load_validation_without_gpu(lib):
    import synth
    import paper_2601_03700_gb300 as adept
    assert lib.adept_status_string(0) == b"ok"
    assert lib.adept_status_string(3) == b"capacity exceeded"
    bad = synth.tiny_config(head_dim=48)
    with pytest.raises(adept.AdeptError) as ei:
        adept.adept_model_load(bad, {})
    assert ei.value.status == 1 and "head_dim" in str(ei.value)
    bad2 = synth.tiny_config(family=1, max_pos=10)
    with pytest.raises(adept.AdeptError) as ei:
        adept.adept_model_load(bad2, {})
    assert "max_pos" in str(ei.value)
    # NULL model handles are rejected, not dereferenced
    assert lib.adept_prefill(None, 1, 1, None, ctypes.c_float(0.5), None, None, None, None, None, None) == 1
    assert lib.adept_set_option(None, 1, 1) == 1
    assert lib.adept_launch_count(None) == 0
    assert lib.adept_hsm_train_init(None, 8, None) == 1
    assert lib.adept_hsm_train_step(None, 1, None, None, None, None, None, None, None) == 1
    assert lib.adept_hsm_train_read(None, 0, 0, None, 0, None) == 1
    assert lib.adept_hsm_train_step_cls(None, 1, None, None, None, None, 0, None, 1.0, None, None, None) == 1
    assert lib.adept_hsm_param_numel(None, 0) == -1
