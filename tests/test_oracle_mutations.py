"""The oracle's pins must catch plausible mistakes.

Each case plants one mistake in a copy of the oracle source (on the CPU),
builds it, and runs the pin tests against that build in a subprocess; the
pins must fail.  The real oracle is never modified.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    "draft node does not see itself": (
        "for (int m = n; m >= 0; m = parents_of_seq[m]) visible[m] = 1;",
        "for (int m = parents_of_seq[n]; m >= 0; m = parents_of_seq[m]) visible[m] = 1;"),
    "chain sees one slot too few": (
        "for (int m = 0; m <= n; ++m) visible[m] = 1;",
        "for (int m = 0; m < n; ++m) visible[m] = 1; visible[n] = 1; if (n > 0) visible[n - 1] = 0;"),
    "page offset off by one": ("j % d->page_size;", "(j + 1) % d->page_size;"),
    "softmax scale dropped": ("s.push_back(scale * dot);", "s.push_back(dot);"),
    "wrong GQA head mapping": ("const int kvh = h / G;", "const int kvh = h % d->hkv;"),
    "RoPE sign flipped": ("y[j + half] = x[j + half] * cs + x[j] * sn;",
                          "y[j + half] = x[j + half] * cs - x[j] * sn;"),
    "RoPE wrong pair": ("y[j] = x[j] * cs - x[j + half] * sn;",
                        "y[j] = x[j] * cs - x[(j + half + 1) % D] * sn;"),
    "lse in base 2": ("const double row_lse = m + std::log(sum);",
                      "const double row_lse = m + std::log2(sum);"),
    "append ignores n0": ("+ n0 + i) * D;", "+ i) * D;"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    src = open(os.path.join(ROOT, "oracle", "kvshot_oracle.cpp")).read()
    before, after = MUTATIONS[name]
    assert before in src, f"mutation site for '{name}' not found"
    shutil.copy(os.path.join(ROOT, "oracle", "kvshot_oracle.h"), tmp_path)
    (tmp_path / "kvshot_oracle.cpp").write_text(src.replace(before, after))
    lib = tmp_path / "libmutant.so"
    subprocess.run(["g++", "-O1", "-std=c++17", "-fPIC", "-shared", "-pthread", "-o", str(lib),
                    str(tmp_path / "kvshot_oracle.cpp")], check=True)
    env = dict(os.environ, KVO_LIB_OVERRIDE=str(lib))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "tests/test_oracle.py", "tests/test_oracle_rope.py"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"pins did not catch: {name}\n{r.stdout[-2000:]}"
