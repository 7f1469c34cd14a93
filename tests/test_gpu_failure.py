"""Failure detection without a GPU fault: a device wait that nothing ever
completes gives up after its time limit, the host reads CG_ERR_TIMEOUT from
the status word, and the device keeps working (the next calls succeed)."""
import numpy as np
import pytest

import seeded_inputs as SI
from tests._cmp import assert_scores_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cg():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19490_gb300 as m
    m.build()
    return m


def test_bounded_wait_times_out_and_device_stays_usable(cg, orc):
    import time
    import torch
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    t0 = time.perf_counter()
    cg.cg_selftest_bounded_wait(20000, st)            # 20 ms limit
    status, word = cg.cg_read_status(st)
    elapsed = time.perf_counter() - t0
    assert status == 6 and word == cg.DEVFLAG_TIMEOUT
    assert 0.015 < elapsed < 5.0
    # the context is intact: a full drift + ranking pass still matches the oracle
    acts, refs = SI.drift_arrays(3, 4, 40000, seed=2)
    st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    g = cg.cg_drift_scores(torch.from_numpy(acts.view(np.float16)).cuda(),
                           torch.from_numpy(refs).cuda(), 3, 4, status=st2).cpu().numpy()
    assert cg.cg_read_status(st2) == (0, 0)
    assert_scores_close(g, orc.drift_scores(acts, refs, 3, 4))


def test_selftest_argument_checks(cg):
    import torch
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    for bad in (0, 10 ** 7 + 1):
        with pytest.raises(cg.CgError):
            cg.cg_selftest_bounded_wait(bad, st)
    assert cg.cg_read_status(st) == (0, 0)
