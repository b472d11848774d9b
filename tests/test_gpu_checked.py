"""The checked build (-DSEMSHARE_CHECKED, include/semshare.h: semshare_checked_build): the same
pipelined calls run with the bookkeeping checks compiled in raise no check, give the same bits as
the plain build, and a check that fails on purpose reaches the error word with its kernel id and
source line."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, os.path.join(ROOT, "tests"))

pytestmark = pytest.mark.gpu


def test_checked_build_raises_no_check_and_matches_plain_build(tmp_path):
    import checked_workload

    import paper_2509_24832_gb300 as ss

    assert not ss.semshare_checked_build()
    out = tmp_path / "checked.npz"
    env = dict(os.environ, SEMSHARE_CHECKED="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "checked_workload.py"), str(out)], env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    checked = dict(np.load(out))
    assert checked.pop("checked")[0] == 1
    low, kernel, line = checked.pop("selftest")
    assert low == ss.FLAG_CHECK and kernel == ss.KERNEL_SELFTEST and line > 0
    plain = checked_workload.run(torch.device("cuda"))
    assert sorted(plain) == sorted(checked)
    for k in plain:
        np.testing.assert_array_equal(plain[k], checked[k], err_msg=k)


def test_plain_build_has_no_selftest():
    import paper_2509_24832_gb300 as ss

    f = ss.new_err_flag()
    with pytest.raises(ss.SemshareError):
        ss.semshare_check_selftest(f)
