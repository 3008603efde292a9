"""Failure detection without a GPU fault: every device-side wait of the
library is bounded; when one gives up, the kernel records it in the
context's error word and exits, the host reports GCPSL_E_TIMEOUT and the
context turns sticky (GCPSL_E_STATE), while the GPU stays usable.  The
wait is made to run out on an mbarrier that nothing arrives on."""
import numpy as np
import pytest

import paper_2609_29395_gb300 as pkg
from paper_2609_29395_gb300 import binding, configs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _ctx():
    w = configs.WORKLOADS["tiny"]
    ds, assign, params = configs.build_inputs(w)
    return pkg.Context(w.arch, w.num_clients, w.num_clusters, assign, w.B, w.F, 4, ds.images,
                       ds.labels, ds.owner, params, bf16=False, lr=w.lr)


def test_bounded_wait_reports_timeout_and_context_turns_sticky():
    ctx = _ctx()
    ctx.step()
    with pytest.raises(binding.GcpslError) as e:
        ctx.check_wait_timeout(1_000_000)           # 1 ms
    assert e.value.status == binding.GCPSL_E_TIMEOUT
    assert "gave up" in str(e.value)
    with pytest.raises(binding.GcpslError) as e:
        ctx.step()
    assert e.value.status == binding.GCPSL_E_STATE
    ctx.close()
    # the GPU is still usable: a fresh context steps normally
    ctx2 = _ctx()
    loss, active = ctx2.step(stats=True)
    assert np.isfinite(loss).all() and (active > 0).all()
    with pytest.raises(binding.GcpslError) as e:
        ctx2.check_wait_timeout(0)                  # outside [1, 1e9]
    assert e.value.status == binding.GCPSL_E_INVAL
    ctx2.step()                                     # a bad argument is not sticky
    ctx2.close()
