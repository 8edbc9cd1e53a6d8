"""The projection oracle's pins must catch plausible mistakes (planted in a copy of oracle/project.py, CPU)."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    "rotation sign flipped": ("[a * c - b * s, b * c + a * s]", "[a * c + b * s, b * c - a * s]"),
    "wrong pair partner": ("a, b = h[..., :HEAD_DIM // 2], h[..., HEAD_DIM // 2:]",
                           "a, b = h[..., :HEAD_DIM // 2], np.roll(h[..., HEAD_DIM // 2:], 1, axis=-1)"),
    "frequency exponent off": ("base ** (-2.0 * j / HEAD_DIM)", "base ** (-1.0 * j / HEAD_DIM)"),
    "RoPE on the values too": ("        kp = rope(kp, np.asarray(positions), rope_base)",
                               "        kp = rope(kp, np.asarray(positions), rope_base)\n        vp = rope(vp, np.asarray(positions), rope_base)"),
    "layers concatenated in reverse": ("kp = k.reshape(T, L * hkv * D) @ wk.T", "kp = k[:, ::-1].reshape(T, L * hkv * D) @ wk.T"),
    "page offset off by one": ("* page_size + (p % page_size)[:, None]", "* page_size + ((p + 1) % page_size)[:, None]"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    src = open(os.path.join(ROOT, "oracle", "project.py")).read()
    before, after = MUTATIONS[name]
    assert before in src, f"mutation site for '{name}' not found"
    mutant = tmp_path / "project_mutant.py"
    mutant.write_text(src.replace(before, after))
    env = dict(os.environ, KVO_PROJECT_OVERRIDE=str(mutant))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "tests/test_oracle_project.py"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode != 0, f"pins did not catch: {name}\n{r.stdout[-2000:]}"
