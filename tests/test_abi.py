"""The C-ABI library loads without a GPU, exports every entry point that
include/ivit.h declares, and rejects bad configurations before touching the device."""
import os
import re
import subprocess

import numpy as np
import pytest

from paper_2607_12287_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def pkg():
    from paper_2607_12287_gb300 import build
    build.build()
    import paper_2607_12287_gb300 as p
    p.load()
    return p


def declared_entry_points():
    text = open(os.path.join(ROOT, "include", "ivit.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ivit_[a-z_]+)\s*\(", text)))


def test_every_entry_point_is_documented_in_the_header():
    # each declaration (or group of adjacent declarations) follows a comment block that
    # states the operation, argument layouts, ownership and errors
    lines = open(os.path.join(ROOT, "include", "ivit.h")).read().splitlines()
    decl = re.compile(r"^[A-Za-z].*\b(ivit_[a-z_]+)\s*\(")
    undocumented = []
    for i, line in enumerate(lines):
        m = decl.match(line)
        if not m:
            continue
        j = i - 1
        # skip earlier declarations of the group (and their continuation lines) and macros
        while j >= 0 and (lines[j].startswith("#define") or lines[j].startswith(" ") and not
                          lines[j].strip().endswith("*/") or decl.match(lines[j])):
            j -= 1
        if j < 0 or not lines[j].rstrip().endswith("*/"):
            undocumented.append(m.group(1))
    assert not undocumented, f"entry points without a comment block: {undocumented}"


def test_header_declares_the_binding_names(pkg):
    assert declared_entry_points() == sorted(pkg.EXPORTED)


def test_library_exports_every_declared_symbol(pkg):
    out = subprocess.run(["nm", "-D", "--defined-only", pkg.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (ivit_[a-z_]+)$", out, flags=re.M))
    missing = set(declared_entry_points()) - exported
    assert not missing, f"missing symbols: {missing}"


def test_weights_size_matches_generator_layout(pkg):
    for shape in (synth.VIT_TINY_224, synth.SO400M_224, synth.SO400M_448):
        assert pkg.ivit_weights_size(pkg.make_config(shape)) == synth.weight_count(shape)


@pytest.mark.parametrize("field,value", [
    ("dim", 100), ("heads", 7), ("patch", 15), ("mlp_dim", 1001), ("depth", 0),
    ("n_views", 0), ("gelu", 5), ("select_mode", 9), ("ref_mode", 3), ("ln_eps", 0.0),
    ("score_source", 2), ("schedule", 4), ("mlp_tokens", 2),
])
def test_bad_config_rejected_before_device_work(pkg, field, value):
    cfg = pkg.make_config(synth.SO400M_224)
    setattr(cfg, field, value)
    assert pkg.ivit_weights_size(cfg) == 0
    with pytest.raises(pkg.IvitError) as e:
        pkg.ivit_create(cfg, np.zeros(8, np.uint16))
    assert e.value.code == pkg.IVIT_ERR_SHAPE
    assert pkg.ivit_last_error(None)


def test_too_many_tokens_rejected(pkg):
    cfg = pkg.make_config(synth.EncoderShape(896, 896, 14, 1152, 1, 16, 4304))  # 4096 tokens
    with pytest.raises(pkg.IvitError) as e:
        pkg.ivit_create(cfg, np.zeros(8, np.uint16))
    assert "1024" in str(e.value)


def test_null_handle_calls_return_arg_error(pkg):
    L = pkg.load()
    assert L.ivit_encode_full(None, None, None, None) == pkg.IVIT_ERR_ARG
    assert L.ivit_encode_incremental(None, None, None, None, None) == pkg.IVIT_ERR_ARG
    assert L.ivit_reset(None, 0) == pkg.IVIT_ERR_ARG
    assert L.ivit_get_changed(None, 0, None, None, None) == pkg.IVIT_ERR_ARG
    assert L.ivit_device_status(None, None) == pkg.IVIT_ERR_ARG
    L.ivit_destroy(None)


C_CLIENT = r"""
#include <stdio.h>
#include <string.h>
#include "ivit.h"

int main(void) {
  ivit_config c;
  memset(&c, 0, sizeof c);
  c.img_h = 224; c.img_w = 224; c.patch = 14; c.dim = 1152; c.depth = 27; c.heads = 16;
  c.mlp_dim = 4304; c.n_streams = 1; c.n_views = 1; c.ln_eps = 1e-6f;
  c.gelu = IVIT_GELU_TANH; c.select_mode = IVIT_SEL_THRESHOLD; c.threshold = 0.98f;
  c.ref_mode = IVIT_REF_PREV_FRAME; c.score_source = IVIT_SCORE_EMBED;
  c.schedule = IVIT_SCHED_INCREMENTAL; c.mlp_tokens = IVIT_MLP_UPDATED;
  printf("%zu\n", ivit_weights_size(&c));
  c.dim = 100; /* not a multiple of 64 */
  ivit_handle* h = (ivit_handle*)0;
  int r = ivit_create(&c, (const uint16_t*)0, &h);
  printf("%d %d %s\n", r, h == (ivit_handle*)0, ivit_last_error((const ivit_handle*)0));
  printf("%d\n", ivit_reset((ivit_handle*)0, 0));
  ivit_destroy((ivit_handle*)0);
  return 0;
}
"""


def test_header_is_plain_c_and_links(pkg, tmp_path):
    # a C99 client compiled against include/ivit.h and linked with the library; it calls
    # only entry points that need no device
    src = tmp_path / "client.c"
    src.write_text(C_CLIENT)
    exe = tmp_path / "client"
    lib_dir = os.path.dirname(pkg.LIB_PATH)
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe), "-L", lib_dir, "-l:libivit.so", f"-Wl,-rpath,{lib_dir}"],
                   check=True, capture_output=True, text=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines()
    assert int(out[0]) == synth.weight_count(synth.SO400M_224)
    code, null_out, msg = out[1].split(" ", 2)
    assert int(code) == pkg.IVIT_ERR_SHAPE and null_out == "1" and "64" in msg
    assert int(out[2]) == pkg.IVIT_ERR_ARG


def test_misaligned_pointers_rejected_before_device_work(pkg):
    # raw addresses: the entry points must turn a misaligned pointer into IVIT_ERR_ARG
    # on the host, before any CUDA call (none can succeed on a machine without a GPU)
    L = pkg.load()
    ok16, off4, odd = 0x10000, 0x10004, 0x10001
    assert L.ivit_select_noalloc(off4, ok16, 1, 16, 8, 0, 0.98, 0, ok16, ok16, None) == pkg.IVIT_ERR_ARG
    assert L.ivit_select_noalloc(ok16, off4, 1, 16, 8, 0, 0.98, 0, ok16, ok16, None) == pkg.IVIT_ERR_ARG
    assert L.ivit_select_noalloc(ok16, ok16, 1, 16, 8, 0, 0.98, 0, odd, ok16, None) == pkg.IVIT_ERR_ARG
    assert L.ivit_select_noalloc(ok16, ok16, 1, 16, 8, 0, 0.98, 0, ok16, odd, None) == pkg.IVIT_ERR_ARG
    assert "aligned" in pkg.ivit_last_error(None)
    for i in range(7):
        ptrs = [ok16] * 7
        ptrs[i] = odd
        x0, v0, v7, al, be, b, xT = ptrs
        assert L.ivit_action_combine(x0, v0, v7, al, be, b, 2, 8, xT, None) == pkg.IVIT_ERR_ARG
