"""The QK-norm oracle's pins must catch plausible mistakes (planted in a copy of oracle/qknorm.py, CPU)."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    "sum instead of mean": ("ms = np.mean(x * x, axis=-1, keepdims=True)", "ms = np.sum(x * x, axis=-1, keepdims=True)"),
    "eps outside the root": ("x / np.sqrt(ms + eps) * w", "x / (np.sqrt(ms) + eps) * w"),
    "no square root": ("x / np.sqrt(ms + eps) * w", "x / (ms + eps) * w"),
    "weights dropped": ("x / np.sqrt(ms + eps) * w", "x / np.sqrt(ms + eps)"),
    "norm over all heads": ("ms = np.mean(x * x, axis=-1, keepdims=True)",
                            "ms = np.mean(x * x, axis=tuple(range(1, x.ndim)), keepdims=True) if x.ndim > 2 else np.mean(x * x, axis=-1, keepdims=True)"),
    "k normalised with the q weights": ("kn = rope(rms_norm(k, wk, eps)", "kn = rope(rms_norm(k, wq, eps)"),
    "weights applied after RoPE": (
        "qn = rope(rms_norm(q, wq, eps).reshape(C * n, hq * D), flat_pos, rope_base).reshape(C, n, hq, D)",
        "qn = rope(rms_norm(q, np.ones(D), eps).reshape(C * n, hq * D), flat_pos, rope_base).reshape(C, n, hq, D) * wq"),
    "values normalised too": ("v.transpose(0, 2, 1, 3).copy()", "rms_norm(v, wk, eps).transpose(0, 2, 1, 3)"),
    "slot axes swapped": ("return qn, kn.transpose(0, 2, 1, 3), v.transpose(0, 2, 1, 3).copy()",
                          "return qn, kn.transpose(0, 2, 1, 3), v.transpose(2, 0, 1, 3).copy()"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    src = open(os.path.join(ROOT, "oracle", "qknorm.py")).read()
    before, after = MUTATIONS[name]
    assert before in src, f"mutation site for '{name}' not found"
    mutant = tmp_path / "qknorm_mutant.py"
    mutant.write_text(src.replace(before, after))
    env = dict(os.environ, KVO_QKNORM_OVERRIDE=str(mutant))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "tests/test_oracle_qknorm.py"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode != 0, f"pins did not catch: {name}\n{r.stdout[-2000:]}"
