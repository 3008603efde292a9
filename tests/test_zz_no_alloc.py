"""The allocation-free round sampler against the context's own sampler.

gcpsl_sample_round_noalloc serves callers that may not allocate device
memory while they run (a plug-in whose host framework owns the device's
memory, or a process that reserves everything up front).  It keeps its
working storage in a fixed array inside the library, so it must return
exactly the batches that gcpsl_step draws, call after call, even though every
call reuses the same storage.  This file is named so that pytest collects it
last.
"""
import numpy as np
import pytest

import paper_2609_29395_gb300 as pkg
from paper_2609_29395_gb300 import configs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def test_noalloc_sampler_matches_gcpsl_step_round_after_round():
    import torch
    w = configs.WORKLOADS["tiny"]
    ds, assign, params = configs.build_inputs(w)
    C, K, B, seed = w.num_clusters, w.num_clients, w.B, 4
    ctx = pkg.Context(w.arch, K, C, assign, B, 0, seed, ds.images, ds.labels, ds.owner, params,
                      bf16=False, lr=w.lr)
    # the clusters' example ids, ascending within each cluster
    ids = [np.flatnonzero(assign[ds.owner] == n).astype(np.int32) for n in range(C)]
    offsets = np.concatenate([[0], np.cumsum([len(x) for x in ids])]).astype(np.int64)
    dev = torch.device("cuda", 0)
    d_ids = torch.from_numpy(np.concatenate(ids)).to(dev)
    d_owner = torch.from_numpy(ds.owner).to(dev)
    d_labels = torch.from_numpy(ds.labels).to(dev)
    d_idx = torch.full((C, B), -1, dtype=torch.int32, device=dev)
    d_counts = torch.full((C, K), -1, dtype=torch.int32, device=dev)
    d_active = torch.full((C,), -1, dtype=torch.int32, device=dev)
    d_blab = torch.full((C, B), -1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream().cuda_stream
    rounds_per_epoch = min(len(x) for x in ids) // B
    # two calls in a row, then on across an epoch boundary
    for t in range(rounds_per_epoch + 2):
        _loss, active = ctx.step(stats=True)
        gi, gc = ctx.sample()
        pkg.binding.gcpsl_sample_round_noalloc(
            d_ids.data_ptr(), offsets, d_owner.data_ptr(), d_labels.data_ptr(), K, C, B, t, 0,
            seed, d_idx.data_ptr(), d_counts.data_ptr(), d_active.data_ptr(), d_blab.data_ptr(),
            stream)
        torch.cuda.synchronize()
        assert (d_idx.cpu().numpy() == gi).all(), t
        assert (d_counts.cpu().numpy() == gc).all(), t
        assert (d_active.cpu().numpy() == active).all(), t
        assert (d_blab.cpu().numpy() == ds.labels[gi]).all(), t
    ctx.close()


def test_noalloc_sampler_rejects_sizes_beyond_its_storage():
    import torch
    dev = torch.device("cuda", 0)
    z = torch.zeros(16, dtype=torch.int32, device=dev)
    big = np.array([0, 300_000], dtype=np.int64)     # more examples than the array holds
    with pytest.raises(pkg.GcpslError) as e:
        pkg.binding.gcpsl_sample_round_noalloc(z.data_ptr(), big, z.data_ptr(), z.data_ptr(), 4,
                                               1, 8, 0, 0, 1, z.data_ptr(), z.data_ptr(),
                                               z.data_ptr(), z.data_ptr())
    assert e.value.status == pkg.binding.GCPSL_E_INVAL
    assert "262144" in str(e.value)
