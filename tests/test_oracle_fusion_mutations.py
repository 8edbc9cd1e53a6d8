"""The fusion oracle's pins must catch plausible mistakes.

Each case plants one mistake in a copy of oracle/fusion.py (on the CPU) and
runs tests/test_oracle_fusion.py against that copy in a subprocess; the pins
must fail.  The real oracle is never modified.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    "gate sees n in place of delta": ("np.concatenate([n, o, delta], axis=1)", "np.concatenate([n, o, n], axis=1)"),
    "gate blocks swapped": ("np.concatenate([n, o, delta], axis=1)", "np.concatenate([o, n, delta], axis=1)"),
    "W_delta transposed": ("delta @ w_delta.T", "delta @ w_delta"),
    "bias dropped": ("sigmoid(x @ w_g.T + b_g)", "sigmoid(x @ w_g.T)"),
    "delta sign flipped": ("delta = o - n", "delta = n - o"),
    "residual taken from o": ("return n + g * (delta @ w_delta.T)", "return o + g * (delta @ w_delta.T)"),
    "gate not squashed": ("g = sigmoid(x @ w_g.T + b_g)", "g = np.tanh(x @ w_g.T + b_g)"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    src = open(os.path.join(ROOT, "oracle", "fusion.py")).read()
    before, after = MUTATIONS[name]
    assert before in src, f"mutation site for '{name}' not found"
    mutant = tmp_path / "fusion_mutant.py"
    mutant.write_text(src.replace(before, after))
    env = dict(os.environ, KVO_FUSION_OVERRIDE=str(mutant))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "tests/test_oracle_fusion.py"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode != 0, f"pins did not catch: {name}\n{r.stdout[-2000:]}"
