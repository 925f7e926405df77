"""The bounded in-kernel waits: a wait that runs out reports PRESTO_DEV_TIMEOUT in
the status word and the kernel returns normally, so the context stays usable.  The
wait here is on a barrier phase that nothing completes, with nothing asynchronous
in flight (presto_selftest_wait_timeout); no GPU fault, trap or hang is involved."""

import numpy as np
import torch

import paper_2607_22634_gb300 as P
from oracle import presto_oracle as O
from gpu_common import GPU

pytestmark = GPU

TIMEOUT = 0x20  # PRESTO_DEV_TIMEOUT


def test_wait_runs_out_reports_timeout_and_returns():
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.presto_selftest_wait_timeout(st, 2_000_000)   # about a millisecond of SM cycles
    torch.cuda.synchronize()
    assert int(st.item()) & TIMEOUT
    # the context still works: an ordinary call right after gives the oracle's answer
    g = torch.Generator().manual_seed(5)
    x = torch.randn(1, 3, 5000, generator=g)
    st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    ids, logq, lse = P.presto_topk(x.cuda(), 4, dev_status=st2)
    torch.cuda.synchronize()
    oids, _, _ = O.topk_logsoftmax(x.reshape(3, 5000).double().numpy(), 4)
    np.testing.assert_array_equal(ids.cpu().numpy().reshape(3, 4), oids)
    assert int(st2.item()) == 0


def test_zero_limit_times_out_at_once():
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.presto_selftest_wait_timeout(st, 0)
    torch.cuda.synchronize()
    assert int(st.item()) & TIMEOUT
