"""The documented usage example (tests/usage_example.py) runs as written: a full resnet18-n8
ADPSGD run, about a second."""
import os
import sys

import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def test_usage_example_runs(capsys):
    sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))
    import usage_example
    stats, t = usage_example.main()
    assert stats.rounds == len(t["k"]) > 0 and stats.sync_step_launches == stats.rounds
    out = capsys.readouterr().out.split()
    assert int(out[0]) == stats.rounds
