"""The e4m3 oracle's pins must catch plausible mistakes (planted in a copy of oracle/fp8.py, CPU)."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    "exponent bias 8": ("np.exp2(e - 7.0)", "np.exp2(e - 8.0)"),
    "subnormals with an implicit one": ("(m / 8.0) * 2.0 ** -6)", "(1.0 + m / 8.0) * 2.0 ** -7)"),
    "no NaN codes": ("return np.where((e == 15) & ((c & 7) == 7), np.nan, val)", "return val"),
    "mantissa over 16": ("(1.0 + m / 8.0) * np.exp2", "(1.0 + m / 16.0) * np.exp2"),
    "sign bit ignored": ("sign = np.where((c >> 7) & 1, -1.0, 1.0)", "sign = 1.0"),
    "scale exponent negated": ("e4m3_value(codes) * 2.0 ** int(scale_exp)", "e4m3_value(codes) * 2.0 ** -int(scale_exp)"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    src = open(os.path.join(ROOT, "oracle", "fp8.py")).read()
    before, after = MUTATIONS[name]
    assert before in src, f"mutation site for '{name}' not found"
    mutant = tmp_path / "fp8_mutant.py"
    mutant.write_text(src.replace(before, after))
    env = dict(os.environ, KVO_FP8_OVERRIDE=str(mutant))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "tests/test_oracle_fp8.py"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode != 0, f"pins did not catch: {name}\n{r.stdout[-2000:]}"
