"""The README's Python examples run as written (in order, one namespace) and
give tables and trajectories of the stated shapes."""
import os
import re

import numpy as np
import pytest

from gpu_util import need_gpu

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_readme_examples_run():
    need_gpu()
    text = open(os.path.join(ROOT, "README.md")).read()
    blocks = re.findall(r"```python\n(.*?)```", text, re.S)
    assert len(blocks) == 2
    ns = {}
    exec(compile(blocks[0], "README-1", "exec"), ns)
    table = ns["table"]
    assert table.shape == (64, 4)
    assert np.all(np.isfinite(table)) and np.all(table[:, 1] > 0)
    assert np.all(np.abs(table[:, 0]) <= 13)
    exec(compile(blocks[1], "README-2", "exec"), ns)
    traj = ns["traj"]
    obs = traj["obs"].cpu().numpy()
    assert obs.shape == (2, 25, 4096, 3, 20)
    act = traj["action"].cpu().numpy()
    assert act.max() <= 4
    done = traj["done"].cpu().numpy()
    assert np.all(done[:, -1] == 1) and np.all(done[:, :-1] == 0)
    assert np.all(traj["reward"].cpu().numpy() <= 0)
