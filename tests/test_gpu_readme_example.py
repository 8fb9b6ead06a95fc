"""The usage example in README.md runs as written (full resnet18-n8 ADPSGD run, about a second)."""
import os
import re

import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_readme_python_example_runs(capsys):
    text = open(os.path.join(ROOT, "README.md")).read()
    blocks = re.findall(r"```python\n(.*?)```", text, flags=re.S)
    assert len(blocks) == 1
    scope = {}
    exec(compile(blocks[0], "README.md", "exec"), scope)
    stats, t = scope["stats"], scope["t"]
    assert stats.rounds == len(t["k"]) > 0 and stats.sync_step_launches == stats.rounds
    out = capsys.readouterr().out.split()
    assert int(out[0]) == stats.rounds
