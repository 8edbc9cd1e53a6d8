"""The C ABI boundary, on the CPU: the library builds, loads and exports every
function include/kvshot.h declares; the Python descriptor mirrors the C
struct byte for byte; invalid arguments are rejected with their status code
before anything touches CUDA."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2604_26412_gb300 import build as kbuild
from paper_2604_26412_gb300 import kvshot

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "kvshot.h")


@pytest.fixture(scope="module")
def lib():
    kbuild.build()
    return kvshot.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(kvshot_\w+)\s*\(", text)))


def test_header_functions_are_exported(lib):
    names = declared_functions()
    assert set(names) == set(kvshot.EXPORTS)
    out = subprocess.run(["nm", "-D", "--defined-only", kbuild.LIB], capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT (kvshot_\w+)", out))
    for n in names:
        assert n in exported, n
        assert hasattr(lib, n)


def test_descriptor_layout_matches_header(tmp_path):
    fields = [f for f, _ in kvshot.AttnDesc._fields_]
    src = ["#include <stdio.h>", "#include <stddef.h>", '#include "kvshot.h"', "int main(void) {",
           'printf("%zu\\n", sizeof(kvshot_attn_desc));']
    src += [f'printf("%zu\\n", offsetof(kvshot_attn_desc, {f}));' for f in fields]
    src += ["return 0; }"]
    c = tmp_path / "layout.c"
    c.write_text("\n".join(src))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.dirname(HEADER), str(c), "-o", str(exe)], check=True)
    vals = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    assert vals[0] == ctypes.sizeof(kvshot.AttnDesc)
    for f, off in zip(fields, vals[1:]):
        assert getattr(kvshot.AttnDesc, f).offset == off, f


def test_status_strings_and_version(lib):
    for code in range(0, 10):
        assert kvshot.status_string(code) and kvshot.status_string(code) != "unknown status"
    assert kvshot.status_string(42) == "unknown status"
    assert kvshot.version() >= 100


def _desc(**kw):
    base = dict(num_caches=2, num_seqs=2, hq=32, hkv=8, n_nodes=8, n_query=4, n_max=8, max_seq_len=64,
                page_size=16, max_pages_per_seq=4, num_pages=8, l_cap=64, tree=True)
    base.update(kw)
    return kvshot.make_desc(**base)


# Fake, suitably aligned device addresses: never dereferenced, because every
# case below fails validation first.
A = 1 << 20


def _attn(d, **ptrs):
    p = dict(q=A, tk=A, tv=A, pt=A, sl=A, dk=A, dv=A, par=A, out=2 * A, lse=3 * A)
    p.update(ptrs)
    return kvshot.draft_attn_status(d, p["q"], p["tk"], p["tv"], p["pt"], p["sl"], p["dk"], p["dv"], p["par"], p["out"],
                                    p["lse"], stream=0)


@pytest.mark.parametrize("kw,code", [
    (dict(num_caches=0), kvshot.KVSHOT_ERR_SHAPE),
    (dict(num_caches=3, num_seqs=2), kvshot.KVSHOT_ERR_SHAPE),
    (dict(num_caches=2048, num_seqs=2048), kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(hq=30, hkv=8), kvshot.KVSHOT_ERR_SHAPE),
    (dict(head_dim=64), kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(n_query=9), kvshot.KVSHOT_ERR_SHAPE),
    (dict(n_nodes=9), kvshot.KVSHOT_ERR_SHAPE),
    (dict(n_nodes=65, n_max=80), kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(page_size=12), kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(page_size=512), kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(page_size=24), kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(page_size=72), kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(num_pages=0), kvshot.KVSHOT_ERR_SHAPE),
    (dict(max_seq_len=-1), kvshot.KVSHOT_ERR_SHAPE),
    (dict(flags=0x80), kvshot.KVSHOT_ERR_SHAPE),
    (dict(flags=0x40), kvshot.KVSHOT_ERR_SHAPE),
    (dict(flags=kvshot.KVSHOT_TARGET_FP8, k_scale_exp=65), kvshot.KVSHOT_ERR_SHAPE),
    (dict(flags=kvshot.KVSHOT_TARGET_FP8, v_scale_exp=-65), kvshot.KVSHOT_ERR_SHAPE),
    # fp8 on the tcgen05 kernel: stacks of up to 128 rows only (160 here: 40 query nodes x G = 4)
    (dict(flags=kvshot.KVSHOT_TARGET_FP8 | kvshot.KVSHOT_FORCE_TC, n_nodes=40, n_query=40, n_max=40),
     kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(flags=kvshot.KVSHOT_TARGET_FP8 | kvshot.KVSHOT_FORCE_CC), kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(flags=kvshot.KVSHOT_FORCE_CC | kvshot.KVSHOT_FORCE_MMA), kvshot.KVSHOT_ERR_SHAPE),
    (dict(flags=kvshot.KVSHOT_FORCE_MMA | kvshot.KVSHOT_FORCE_TC), kvshot.KVSHOT_ERR_SHAPE),
    (dict(flags=kvshot.KVSHOT_FORCE_TC, hq=24, hkv=8), kvshot.KVSHOT_ERR_UNSUPPORTED),
    (dict(num_ctas=-1), kvshot.KVSHOT_ERR_SHAPE),
    (dict(scale=float("inf")), kvshot.KVSHOT_ERR_SHAPE),
    (dict(scale=-0.5), kvshot.KVSHOT_ERR_SHAPE),        # a softmax scale is positive (0 = default)
])
def test_invalid_descriptor_codes(lib, kw, code):
    assert _attn(_desc(**kw)) == code
    if "page_size" not in kw and "num_pages" not in kw:
        assert kvshot.workspace_size(_desc(**kw)) == 0


def test_null_and_alignment_codes(lib):
    assert kvshot.draft_attn_status(None, A, A, A, A, A, A, A, A, A, A, stream=0) == kvshot.KVSHOT_ERR_NULL
    d = _desc()
    assert _attn(d, q=None) == kvshot.KVSHOT_ERR_NULL
    assert _attn(d, par=None) == kvshot.KVSHOT_ERR_NULL        # tree needs parents
    assert _attn(d, sl=None) == kvshot.KVSHOT_ERR_NULL
    assert _attn(d, q=A + 8) == kvshot.KVSHOT_ERR_ALIGN
    assert _attn(d, tk=A + 2) == kvshot.KVSHOT_ERR_ALIGN
    assert _attn(d, lse=A + 2) == kvshot.KVSHOT_ERR_ALIGN
    assert _attn(d, out=A + 4) == kvshot.KVSHOT_ERR_ALIGN
    assert _attn(_desc(l_cap=0), pt=None) == kvshot.KVSHOT_ERR_SHAPE   # contiguous layout needs l_cap
    assert _attn(_desc(n_query=0)) == kvshot.KVSHOT_OK                  # no-op


def test_append_argument_codes(lib):
    d = _desc()
    call = lambda **k: kvshot.draft_append_status(d, k.get("q", A), k.get("k", A), k.get("v", A), k.get("pos", A),
                                                  k.get("n0", 0), k.get("n_new", 2), k.get("base", 1e6), A, A,
                                                  k.get("qo", 2 * A), stream=0)
    assert kvshot.draft_append_status(None, A, A, A, A, 0, 1, 1e6, A, A, A, stream=0) == kvshot.KVSHOT_ERR_NULL
    assert call(n0=7, n_new=2) == kvshot.KVSHOT_ERR_SHAPE
    assert call(n0=-1) == kvshot.KVSHOT_ERR_SHAPE
    assert call(base=0.0) == kvshot.KVSHOT_ERR_SHAPE
    assert call(n_new=0) == kvshot.KVSHOT_OK
    assert call(q=None) == kvshot.KVSHOT_ERR_NULL
    assert call(k=A + 4) == kvshot.KVSHOT_ERR_ALIGN
    assert call(pos=A + 2) == kvshot.KVSHOT_ERR_ALIGN
    assert call(qo=A + 256) == kvshot.KVSHOT_ERR_SHAPE                 # partial overlap of q_out and q_in
    assert kvshot.draft_append_status(_desc(head_dim=96), A, A, A, A, 0, 1, 1e6, A, A, A, stream=0) == \
        kvshot.KVSHOT_ERR_UNSUPPORTED


def test_append_qknorm_argument_codes(lib):
    d = _desc()
    call = lambda **k: kvshot.draft_append_qknorm_status(
        k.get("d", d), A, A, A, A, k.get("n0", 0), k.get("n_new", 2), 1e6, k.get("wq", A), k.get("wk", A),
        k.get("eps", 1e-6), A, A, 2 * A, stream=0)
    assert call(d=None) == kvshot.KVSHOT_ERR_NULL
    assert call(eps=0.0) == kvshot.KVSHOT_ERR_SHAPE
    assert call(eps=-1e-6) == kvshot.KVSHOT_ERR_SHAPE
    assert call(eps=float("nan")) == kvshot.KVSHOT_ERR_SHAPE
    assert call(wq=None) == kvshot.KVSHOT_ERR_NULL
    assert call(wk=None) == kvshot.KVSHOT_ERR_NULL
    assert call(wq=A + 2) == kvshot.KVSHOT_ERR_ALIGN
    assert call(wk=A + 2) == kvshot.KVSHOT_ERR_ALIGN
    assert call(n0=7) == kvshot.KVSHOT_ERR_SHAPE          # the plain append's checks apply too
    assert call(n_new=0) == kvshot.KVSHOT_OK
    assert call(d=_desc(head_dim=96)) == kvshot.KVSHOT_ERR_UNSUPPORTED


def test_fusion_descriptor_layout_matches_header(tmp_path):
    fields = [f for f, _ in kvshot.FusionDesc._fields_]
    src = ["#include <stdio.h>", "#include <stddef.h>", '#include "kvshot.h"', "int main(void) {",
           'printf("%zu\\n", sizeof(kvshot_fusion_desc));']
    src += [f'printf("%zu\\n", offsetof(kvshot_fusion_desc, {f}));' for f in fields]
    src += ["return 0; }"]
    c = tmp_path / "layout_fusion.c"
    c.write_text("\n".join(src))
    exe = tmp_path / "layout_fusion"
    subprocess.run(["gcc", "-I", os.path.dirname(HEADER), str(c), "-o", str(exe)], check=True)
    vals = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    assert vals[0] == ctypes.sizeof(kvshot.FusionDesc)
    for f, off in zip(fields, vals[1:]):
        assert getattr(kvshot.FusionDesc, f).offset == off, f


def test_fusion_argument_codes(lib):
    """Every case fails validation (or is the T = 0 no-op) before anything is launched."""
    T, D = 4, 256
    ws = 16 * T * D

    def call(desc, **k):
        return kvshot.gated_delta_status(desc, k.get("n", A), k.get("o", A), k.get("wg", 2 * A), k.get("bg", 3 * A),
                                         k.get("wd", 4 * A), k.get("h", 5 * A), stream=0)

    good = kvshot.make_fusion_desc(num_tokens=T, hidden=D, workspace=6 * A, workspace_bytes=ws)
    assert kvshot.gated_delta_workspace_size(good) == ws
    assert call(None) == kvshot.KVSHOT_ERR_NULL
    assert call(kvshot.make_fusion_desc(num_tokens=-1, hidden=D)) == kvshot.KVSHOT_ERR_SHAPE
    assert call(kvshot.make_fusion_desc(num_tokens=T, hidden=0)) == kvshot.KVSHOT_ERR_SHAPE
    assert call(kvshot.make_fusion_desc(num_tokens=T, hidden=200)) == kvshot.KVSHOT_ERR_UNSUPPORTED
    assert call(kvshot.make_fusion_desc(num_tokens=T, hidden=65536)) == kvshot.KVSHOT_ERR_UNSUPPORTED
    assert kvshot.gated_delta_workspace_size(kvshot.make_fusion_desc(num_tokens=T, hidden=200)) == 0
    assert call(good, n=None) == kvshot.KVSHOT_ERR_NULL
    assert call(good, wd=None) == kvshot.KVSHOT_ERR_NULL
    assert call(good, n=A + 8) == kvshot.KVSHOT_ERR_ALIGN
    assert call(good, wg=2 * A + 4) == kvshot.KVSHOT_ERR_ALIGN
    assert call(good, h=5 * A + 2) == kvshot.KVSHOT_ERR_ALIGN
    assert call(kvshot.make_fusion_desc(num_tokens=T, hidden=D, workspace=6 * A, workspace_bytes=ws - 1)) == \
        kvshot.KVSHOT_ERR_WORKSPACE
    assert call(kvshot.make_fusion_desc(num_tokens=T, hidden=D, workspace=6 * A + 16, workspace_bytes=ws)) == \
        kvshot.KVSHOT_ERR_WORKSPACE
    assert call(kvshot.make_fusion_desc(num_tokens=0, hidden=D)) == kvshot.KVSHOT_OK  # no-op


def test_project_descriptor_layout_matches_header(tmp_path):
    fields = [f for f, _ in kvshot.ProjectDesc._fields_]
    src = ["#include <stdio.h>", "#include <stddef.h>", '#include "kvshot.h"', "int main(void) {",
           'printf("%zu\\n", sizeof(kvshot_project_desc));']
    src += [f'printf("%zu\\n", offsetof(kvshot_project_desc, {f}));' for f in fields]
    src += ["return 0; }"]
    c = tmp_path / "layout_project.c"
    c.write_text("\n".join(src))
    exe = tmp_path / "layout_project"
    subprocess.run(["gcc", "-I", os.path.dirname(HEADER), str(c), "-o", str(exe)], check=True)
    vals = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    assert vals[0] == ctypes.sizeof(kvshot.ProjectDesc)
    for f, off in zip(fields, vals[1:]):
        assert getattr(kvshot.ProjectDesc, f).offset == off, f


def test_project_argument_codes(lib):
    """Every case fails validation (or is the T = 0 no-op) before anything is launched."""
    base = dict(num_tokens=4, num_layers=3, hkv=8, num_caches=2, page_size=16, max_pages_per_seq=4, num_pages=8)
    ws = 2 * 3 * 4 * 8 * 128 * 4

    def desc(**kw):
        b = dict(base, workspace=7 * A, workspace_bytes=ws)
        b.update(kw)
        return kvshot.make_project_desc(**b)

    def call(d, **k):
        return kvshot.kv_project_status(d, k.get("k", A), k.get("v", 2 * A), k.get("wk", 3 * A), k.get("wv", 4 * A),
                                        k.get("tc", 5 * A), k.get("pos", 5 * A + 256), k.get("pt", 6 * A),
                                        k.get("ko", 8 * A), k.get("vo", 9 * A), stream=0)

    assert kvshot.kv_project_workspace_size(desc()) == ws
    assert call(None) == kvshot.KVSHOT_ERR_NULL
    assert call(desc(num_layers=0)) == kvshot.KVSHOT_ERR_SHAPE
    assert call(desc(num_layers=9)) == kvshot.KVSHOT_ERR_UNSUPPORTED
    assert call(desc(head_dim=64)) == kvshot.KVSHOT_ERR_UNSUPPORTED
    assert call(desc(rope_base=0.0)) == kvshot.KVSHOT_ERR_SHAPE
    assert call(desc(num_pages=0)) == kvshot.KVSHOT_ERR_SHAPE
    assert call(desc(), pt=None) == kvshot.KVSHOT_ERR_SHAPE   # contiguous needs l_cap
    assert call(desc(), k=None) == kvshot.KVSHOT_ERR_NULL
    assert call(desc(), tc=None) == kvshot.KVSHOT_ERR_NULL
    assert call(desc(), k=A + 8) == kvshot.KVSHOT_ERR_ALIGN
    assert call(desc(), pos=5 * A + 2) == kvshot.KVSHOT_ERR_ALIGN
    assert call(desc(workspace_bytes=ws - 1)) == kvshot.KVSHOT_ERR_WORKSPACE
    assert call(desc(num_tokens=0)) == kvshot.KVSHOT_OK
    d = desc()
    d.flags = 0x2
    assert call(d) == kvshot.KVSHOT_ERR_SHAPE
