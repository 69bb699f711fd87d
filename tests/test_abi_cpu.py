"""The C-ABI library builds, loads and exports every entry point that
include/vie_head.h declares; host-side argument checks answer with status
codes before any CUDA call (no GPU needed for these paths)."""
import ctypes
import os
import re

import pytest

import paper_2608_27460_gb300 as vie

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "vie_head.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(vie_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    return vie.load()


def test_header_declares_the_binding_exports():
    assert declared_functions() == sorted(vie.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_header_is_plain_c():
    import subprocess
    src = '#include "vie_head.h"\nint main(void){vie_head_props p; (void)p; return VIE_OK;}\n'
    r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.dirname(HEADER),
                        "-x", "c", "-", "-fsyntax-only"], input=src, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_create_rejects_bad_arguments_on_host(lib):
    st, h = vie.vie_head_create(0, 10, 8)
    assert st == vie.VIE_ERR_INVALID_ARG and h is None
    assert "NULL" in vie.vie_last_error()
    fake = 0x10000
    assert vie.vie_head_create(fake, 0, 8)[0] == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_create(fake, 2 ** 31, 8)[0] == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_create(fake, 10, 0)[0] == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_create(fake, 10, vie.VIE_D_MAX + 1)[0] == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_create(fake, 10, 8, dtype=7)[0] == vie.VIE_ERR_UNSUPPORTED
    assert vie.vie_head_create(fake + 1, 10, 8)[0] == vie.VIE_ERR_INVALID_ARG
    out_null = lib.vie_head_create(fake, 10, 8, 0, None)
    assert out_null == vie.VIE_ERR_INVALID_ARG


def test_calls_on_null_handle_are_rejected(lib):
    assert vie.vie_head_destroy(0) == vie.VIE_OK
    assert vie.vie_head_topk(0, 16, 1, 1, 16, 16) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_get_props(0)[0] == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_device_status(0) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_topk_host(0, 16, 1, 1, 16, 16) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_plan(0, 1, 1)[0] == vie.VIE_ERR_INVALID_ARG


def test_scatter_rejects_bad_arguments_on_host(lib):
    p = 0x10000
    assert vie.vie_scatter_sparse_logits(0, p, 1, 1, 8, p) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_scatter_sparse_logits(p, p, 0, 1, 8, p) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_scatter_sparse_logits(p, p, 1, 0, 8, p) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_scatter_sparse_logits(p, p, 1, 1, 0, p) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_scatter_sparse_logits(p, p, 2, 1, 2 ** 62, p) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_scatter_sparse_logits(p + 2, p, 1, 1, 8, p) == vie.VIE_ERR_INVALID_ARG


def test_sampling_rejects_bad_arguments_on_host(lib):
    p = 0x10000
    ok = dict(temperature=1.0, top_p=1.0, min_p=0.0)
    def call(idx=p, logits=p, batch=1, k=50, out_token=p, out_prob=p, **kw):
        a = dict(ok, **kw)
        return vie.vie_sample_topk(idx, logits, batch, k, a["temperature"], a["top_p"], a["min_p"],
                                   0, 0, out_token, out_prob)
    assert call(idx=0) == vie.VIE_ERR_INVALID_ARG
    assert call(out_prob=0) == vie.VIE_ERR_INVALID_ARG
    assert call(batch=0) == vie.VIE_ERR_INVALID_ARG
    assert call(k=0) == vie.VIE_ERR_INVALID_ARG
    assert call(k=vie.VIE_K_MAX + 1) == vie.VIE_ERR_INVALID_ARG
    assert call(temperature=0.0) == vie.VIE_ERR_INVALID_ARG
    assert call(temperature=float("inf")) == vie.VIE_ERR_INVALID_ARG
    assert call(top_p=0.0) == vie.VIE_ERR_INVALID_ARG
    assert call(top_p=1.5) == vie.VIE_ERR_INVALID_ARG
    assert call(min_p=-0.1) == vie.VIE_ERR_INVALID_ARG
    assert call(min_p=1.1) == vie.VIE_ERR_INVALID_ARG
    assert call(logits=p + 2) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_topk_sample(0, p, 1, 50, 1.0, 1.0, 0.0, 0, 0, p, p, 0, p, p) == vie.VIE_ERR_INVALID_ARG


def test_limits_match_the_header():
    text = open(HEADER).read()
    for name in ("VIE_K_MAX", "VIE_BATCH_MAX", "VIE_D_MAX", "VIE_MANY_MAX", "VIE_RECALL_N_MAX",
                 "VIE_RECALL_M_MAX"):
        m = re.search(r"#define\s+" + name + r"\s+(\S+(?:\s*<<\s*\d+\))?)", text)
        assert m, name
        assert eval(m.group(1)) == getattr(vie, name), name


def test_recall_rejects_bad_arguments_on_host(lib):
    p = 0x10000
    def call(exact=p, k=2, approx=p, m=2, n=4, out=p):
        return vie.vie_recall_hits(exact, k, approx, m, n, out)
    assert call(exact=0) == vie.VIE_ERR_INVALID_ARG
    assert call(approx=0) == vie.VIE_ERR_INVALID_ARG
    assert call(out=0) == vie.VIE_ERR_INVALID_ARG
    assert call(n=0) == vie.VIE_ERR_INVALID_ARG
    assert call(n=vie.VIE_RECALL_N_MAX + 1) == vie.VIE_ERR_INVALID_ARG
    assert call(k=0) == vie.VIE_ERR_INVALID_ARG
    assert call(k=vie.VIE_K_MAX + 1) == vie.VIE_ERR_INVALID_ARG
    assert call(m=0) == vie.VIE_ERR_INVALID_ARG
    assert call(m=vie.VIE_RECALL_M_MAX + 1) == vie.VIE_ERR_INVALID_ARG
    assert call(approx=p + 2) == vie.VIE_ERR_INVALID_ARG
    assert "vie_recall_hits" in vie.vie_last_error()
    assert vie.vie_head_topk_many(0, p, 10, 2, p, p) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_topk_many(0, p, 0, 2, p, p) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_head_topk_many(0, p, vie.VIE_MANY_MAX + 1, 2, p, p) == vie.VIE_ERR_INVALID_ARG


def test_product_path_does_not_import_the_oracle():
    pkg = os.path.join(ROOT, "paper_2608_27460_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b", text, re.M), f
                assert "oracle.c" not in text and "liboracle" not in text, f


def test_launch_options_hook(lib):
    """The launch options are set only through the explicit hook: defaults
    as documented, out-of-range values rejected (the option keeps its value),
    VIE_OPT_DEFAULT restores, the context manager puts values back; the
    library reads no environment variable."""
    defaults = {vie.VIE_OPT_STAGE_MIN_KB: 48, vie.VIE_OPT_STATIC_PCT: 85, vie.VIE_OPT_POOL_DIV: 1,
                vie.VIE_OPT_TC_MIN_BATCH: 2, vie.VIE_OPT_TC_KPS: 4, vie.VIE_OPT_TC_MIN_BATCH_E4M3: 1,
                vie.VIE_OPT_HALF_ROWS: -1, vie.VIE_OPT_HOST_H_DIRECT: 1, vie.VIE_OPT_EARLY_MERGE: 1}
    assert len(defaults) == vie.VIE_OPT_COUNT
    for o, v in defaults.items():
        assert vie.vie_get_launch_option(o) == (vie.VIE_OK, v)
    assert vie.vie_set_launch_option(vie.VIE_OPT_STATIC_PCT, 101) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_set_launch_option(vie.VIE_OPT_HALF_ROWS, -2) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_set_launch_option(vie.VIE_OPT_TC_KPS, 0) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_set_launch_option(vie.VIE_OPT_COUNT, 1) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_set_launch_option(-1, 1) == vie.VIE_ERR_INVALID_ARG
    assert vie.vie_get_launch_option(vie.VIE_OPT_STATIC_PCT) == (vie.VIE_OK, 85)
    assert vie.vie_set_launch_option(vie.VIE_OPT_STATIC_PCT, 50) == vie.VIE_OK
    assert vie.vie_get_launch_option(vie.VIE_OPT_STATIC_PCT) == (vie.VIE_OK, 50)
    assert vie.vie_set_launch_option(vie.VIE_OPT_STATIC_PCT, vie.VIE_OPT_DEFAULT) == vie.VIE_OK
    assert vie.vie_get_launch_option(vie.VIE_OPT_STATIC_PCT) == (vie.VIE_OK, 85)
    with vie.launch_options({vie.VIE_OPT_HALF_ROWS: 1, vie.VIE_OPT_TC_MIN_BATCH: 1000}):
        assert vie.vie_get_launch_option(vie.VIE_OPT_HALF_ROWS) == (vie.VIE_OK, 1)
        assert vie.vie_get_launch_option(vie.VIE_OPT_TC_MIN_BATCH) == (vie.VIE_OK, 1000)
    for o, v in defaults.items():
        assert vie.vie_get_launch_option(o) == (vie.VIE_OK, v)
    for src in ("vie_head.cu", "vie_tc_topk.cu", "vie_tc_topk_e4m3.cu", "vie_sample.cu", "vie_recall.cu"):
        text = open(os.path.join(ROOT, "paper_2608_27460_gb300", "csrc", src)).read()
        assert "getenv" not in text, src
