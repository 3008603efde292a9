"""GPU parity: the CUDA library against the CPU oracle on the same seeded
inputs, through the C ABI.

Per round, both sides start from the same state: the oracle's parameters and
momentum (rounded to fp32) are loaded into the GPU context (data flows from
the oracle to the GPU, never back).  Then both take the round and we compare:

* sampler indices, per-client counts and |A| -- bit-exact;
* per-cluster loss -- within 1e-2 absolute;
* cut activation, updated parameters and the update itself (all replicas)
  -- relative L2 < 2e-2;
* every max-pool decision of the GPU -- equal to the oracle's where the
  oracle's window has a unique maximum (no other position within tol times
  the layer's RMS pre-activation), and one of the oracle's valid maxima where
  it has not;
* cut gradient -- relative L2 < 2e-2 over the whole [C][B] tensor (>= 128
  examples per round).

bf16 workloads are compared with the oracle in its bf16-operand mode (same
rounding points, fp64 accumulation).  Tolerances for the fp32 workload are
tighter (stated in that test).
"""
import numpy as np
import pytest

import oracle
import paper_2609_29395_gb300 as pkg
from paper_2609_29395_gb300 import clustering, configs, synth

pytestmark = pytest.mark.gpu

REL_L2 = 2e-2
LOSS_ABS = 1e-2
FUSE_REL = 1e-6


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def rel_l2(a, b):
    a = np.asarray(a, np.float64).ravel()
    b = np.asarray(b, np.float64).ravel()
    return np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30)


def pooled_layers(arch):
    spec = synth.ARCHS[arch]
    convs = spec["client"] + spec["server"]
    return [(i, cout * (h // 2) * (w // 2)) for i, (_ci, cout, h, w, p) in enumerate(convs) if p]


# Gap, in units of the layer's RMS pre-activation, under which two values of a
# max-pool window are both valid maxima.  With bf16 operands a stored activation is exact only to 2^-9
# relative, and a few bf16 rounding decisions upstream can go either way
# (their fp32 and fp64 pre-images straddle a rounding midpoint), so values
# within ~2.5 bf16 ulps (1%) of the maximum are indistinguishable; fp32
# arithmetic leaves only accumulation-order differences.
DECISION_TOL = {True: 1e-2, False: 1e-4}


def pair(arch, K, C, assign, B, F, ds, params, bf16, seed=4, **kw):
    gpu = pkg.Context(arch, K, C, assign, B, F, seed, ds.images, ds.labels, ds.owner, params,
                      bf16=bf16, **kw)
    orc = oracle.Oracle(arch, K, C, assign, B, F, seed, ds.images, ds.labels, ds.owner, params,
                        bf16=bf16, **kw)
    orc.set_tie_tol(DECISION_TOL[bf16])
    return gpu, orc


def load_oracle_state(gpu, orc):
    """Give both sides the oracle's state, rounded to fp32."""
    for n in range(orc.C):
        th = orc.all_params(n).astype(np.float32)
        v = orc.momentum(n).astype(np.float32)
        orc.set_params(n, th.astype(np.float64))
        orc.set_momentum(n, v.astype(np.float64))
        gpu.set_params(n, th)
        gpu.set_momentum(n, v)


def check_decisions(gpu, orc, arch, gpu_clusters=None):
    """Every GPU max-pool decision is a valid maximum of the oracle's window;
    returns the fraction of windows whose decision was unique."""
    uniq_total, n_total = 0, 0
    for layer, per in pooled_layers(arch):
        code = gpu.pool_codes(layer, per)
        if gpu_clusters is not None:
            code = code[gpu_clusters]
        cand = orc.pool_cand(layer)
        pos = (cand & 16) != 0
        amb_sign = (cand & 32) != 0
        arg = code & 3
        chosen_ok = ((cand >> arg) & 1) == 1
        gpu_pos = (code & 4) != 0
        bad_pos = pos & ~amb_sign & ~(gpu_pos & chosen_ok)
        bad_neg = ~pos & ~amb_sign & gpu_pos
        assert not bad_pos.any(), f"layer {layer}: {bad_pos.sum()} invalid max-pool decisions"
        assert not bad_neg.any(), f"layer {layer}: {bad_neg.sum()} invalid ReLU decisions"
        single = np.isin(cand & 15, (1, 2, 4, 8))
        uniq_total += (pos & ~amb_sign & single).sum()
        n_total += (pos & ~amb_sign).sum()
    return uniq_total / max(n_total, 1)


def check_round(gpu, orc, arch, tol=REL_L2, loss_tol=LOSS_ABS, fwd_tol=REL_L2, grad=True):
    """One round from the oracle's state on both sides, then every check.
    The cut-gradient bar is applied to the whole [C][B] tensor: a max-pool
    window whose two largest values are closer than the two sides' rounding
    differences may route its gradient either way (both valid, checked by
    check_decisions), which moves a few examples' gradients; over >= 128
    examples such routings stay well inside the bar.  `grad=False` skips that
    aggregate for tiny batches (the decisions are still checked)."""
    load_oracle_state(gpu, orc)
    before = [orc.all_params(n) for n in range(orc.C)]
    loss, active = gpu.step(stats=True)
    orc.step()
    gi, gc = gpu.sample()
    oi, oc = orc.sample()
    assert (gi == oi).all(), "sample indices differ"
    assert (gc == oc).all(), "per-client counts differ"
    ol, oa = orc.stats()
    assert (active == oa).all()
    assert np.abs(loss - ol).max() < loss_tol, (loss, ol)
    g = gpu.cut(pkg.binding.GCPSL_CUT_ACT)
    assert rel_l2(g, orc.cut(0).reshape(g.shape)) < fwd_tol
    assert check_decisions(gpu, orc, arch) > 0.9
    e = 0.0
    if grad:
        g = gpu.cut(pkg.binding.GCPSL_CUT_GRAD)
        e = rel_l2(g, orc.cut(1).reshape(g.shape))
        assert e < tol, ("cut grad", e)
    worst = 0.0
    for n in range(gpu.C):
        gp, op = gpu.all_params(n), orc.all_params(n)
        assert rel_l2(gp, op) < tol, ("params", n)
        worst = max(worst, rel_l2(gp - before[n], op - before[n]))   # the update itself
    assert worst < tol, ("update", worst)
    return e, worst


def test_tiny_fp32_ten_rounds_with_fusion_and_epoch_rollover():
    """Tiny workload (fp32): 10 rounds, fusion after rounds 5 and 10, an
    epoch boundary at round 8 (n_c / B = 8).  fp32 bars: loss 1e-4, cut
    activation 1e-5, cut gradient, parameters and update 1e-3."""
    w = configs.WORKLOADS["tiny"]
    ds, assign, params = configs.build_inputs(w)
    gpu, orc = pair(w.arch, w.num_clients, w.num_clusters, assign, w.B, w.F, ds, params, False,
                    lr=w.lr, momentum=w.momentum)
    for t in range(w.steps):
        check_round(gpu, orc, w.arch, tol=1e-3, loss_tol=1e-4, fwd_tol=1e-5)
    assert gpu.rounds == w.steps
    assert (gpu.all_params(0) == gpu.all_params(1)).all()   # fused after round 10


def _splitcnn_small(C=2, n=2048, K=32, alpha=0.3, seed=0):
    ds = synth.make_dataset(n, 10, K, alpha, balanced=False, seed_data=seed, seed_split=seed + 1)
    assign = clustering.random_clustering(K, C, seed + 2)
    return ds, assign, synth.init_params(synth.ARCH_SPLIT_CNN)


def test_splitcnn_bf16_rounds_with_fusion():
    """SplitCNN, bf16 operands, C=4 x B=32, fusion every 2 rounds."""
    ds, assign, params = _splitcnn_small(C=4, n=4096)
    gpu, orc = pair(synth.ARCH_SPLIT_CNN, 32, 4, assign, 32, 2, ds, params, True, lr=0.05,
                    momentum=0.9)
    for _ in range(4):
        check_round(gpu, orc, synth.ARCH_SPLIT_CNN)


def test_client_average_rounds_bf16_and_fp32():
    """The per-client average (client_average = 1): the cut gradient scaled by
    B / (|A| b_k) per example before the client backward, on the bf16
    tensor-core path (SplitCNN) and the fp32 path (the 512-image workload);
    the usual bars against the oracle with the same flag, and the client
    update differs from the example-weighted one."""
    ds, assign, params = _splitcnn_small(C=4, n=4096)
    kw = dict(lr=0.05, momentum=0.9, client_average=True)
    gpu, orc = pair(synth.ARCH_SPLIT_CNN, 32, 4, assign, 32, 2, ds, params, True, **kw)
    for _ in range(3):
        check_round(gpu, orc, synth.ARCH_SPLIT_CNN)
    plain = pkg.Context(synth.ARCH_SPLIT_CNN, 32, 4, assign, 32, 2, 4, ds.images, ds.labels,
                        ds.owner, params, lr=0.05, momentum=0.9)
    avg = pkg.Context(synth.ARCH_SPLIT_CNN, 32, 4, assign, 32, 2, 4, ds.images, ds.labels,
                      ds.owner, params, **kw)
    plain.step()
    avg.step()
    pc = plain.P_client
    assert not np.array_equal(plain.all_params(0)[:pc], avg.all_params(0)[:pc])
    np.testing.assert_array_equal(plain.all_params(0)[pc:], avg.all_params(0)[pc:])
    plain.close()
    avg.close()
    w = configs.WORKLOADS["tiny"]
    ds, assign, params = configs.build_inputs(w)
    gpu, orc = pair(w.arch, w.num_clients, w.num_clusters, assign, w.B, w.F, ds, params, False,
                    lr=w.lr, momentum=w.momentum, client_average=True)
    for _ in range(3):
        check_round(gpu, orc, w.arch, tol=1e-3, loss_tol=1e-4, fwd_tol=1e-5)


def test_augmented_rounds_bf16_and_fp32():
    """The crop + flip augmentation of Section V-A fused into the gather (the
    bf16 path's im2col gather and the fp32 path's gather): every round's
    batch is the oracle's augmented batch, so the usual bars hold; and the
    round differs from the unaugmented one."""
    ds, assign, params = _splitcnn_small(C=4, n=4096)
    kw = dict(lr=0.05, momentum=0.9, augment=True)
    gpu, orc = pair(synth.ARCH_SPLIT_CNN, 32, 4, assign, 32, 2, ds, params, True, **kw)
    for _ in range(3):
        check_round(gpu, orc, synth.ARCH_SPLIT_CNN)
    plain = pkg.Context(synth.ARCH_SPLIT_CNN, 32, 4, assign, 32, 2, 4, ds.images, ds.labels,
                        ds.owner, params, lr=0.05, momentum=0.9)
    aug = pkg.Context(synth.ARCH_SPLIT_CNN, 32, 4, assign, 32, 2, 4, ds.images, ds.labels,
                      ds.owner, params, **kw)
    plain.step()
    aug.step()
    assert (plain.sample()[0] == aug.sample()[0]).all()
    assert not np.array_equal(plain.cut(pkg.binding.GCPSL_CUT_ACT), aug.cut(pkg.binding.GCPSL_CUT_ACT))
    plain.close()
    aug.close()
    w = configs.WORKLOADS["tiny"]
    ds, assign, params = configs.build_inputs(w)
    gpu, orc = pair(w.arch, w.num_clients, w.num_clusters, assign, w.B, w.F, ds, params, False,
                    lr=w.lr, momentum=w.momentum, augment=True)
    for _ in range(3):
        check_round(gpu, orc, w.arch, tol=1e-3, loss_tol=1e-4, fwd_tol=1e-5)


def test_epoch_schedule_with_fusion_barrier():
    """F = -1 (Section IV-C): clusters of unequal size take r_n local rounds
    per system epoch of R = max r_n rounds and wait at the fusion barrier
    (no update, loss and |A| 0), then all replicas are fused; the GPU matches
    the oracle round by round through one system epoch and into the next."""
    ds = synth.make_dataset(3072, 10, 24, 0.3, balanced=False, seed_data=2, seed_split=3)
    assign = (np.arange(24) % 6 > 2).astype(np.int32) + (np.arange(24) % 6 > 4).astype(np.int32)
    params = synth.init_params(synth.ARCH_SPLIT_CNN)
    B = 64
    r = np.bincount(assign[ds.owner], minlength=3) // B
    R = int(r.max())
    assert len(set(r.tolist())) == 3 and R <= 24, r
    gpu, orc = pair(synth.ARCH_SPLIT_CNN, 24, 3, assign, B, -1, ds, params, True, lr=0.05,
                    momentum=0.9)
    for t in range(R + 2):
        check_round(gpu, orc, synth.ARCH_SPLIT_CNN)
        active = orc.stats()[1]                 # equal to the GPU's (check_round)
        for n in range(3):
            assert (active[n] == 0) == (t % R >= r[n])
        if t == R - 1:
            assert all((gpu.all_params(n) == gpu.all_params(0)).all() for n in range(3))


def test_client_average_with_waiting_clusters():
    """The per-client average under the epoch schedule: a cluster waiting at
    the fusion barrier still computes its round (not applied), with the
    factor B / (|A| b_k) of its own batch, as the oracle does."""
    ds = synth.make_dataset(768, 10, 12, 0.3, balanced=False, seed_data=4, seed_split=5)
    assign = (np.arange(12) % 3 == 0).astype(np.int32)
    params = synth.init_params(synth.ARCH_SPLIT_CNN)
    B = 64
    r = np.bincount(assign[ds.owner], minlength=2) // B
    assert r.min() < r.max() <= 12, r
    gpu, orc = pair(synth.ARCH_SPLIT_CNN, 12, 2, assign, B, -1, ds, params, True, lr=0.05,
                    momentum=0.9, client_average=True)
    for t in range(int(r.max())):
        # the scaled cut gradient is compared below with the factor divided
        # out: a factor up to B / |A| on a client with one example would let
        # one valid tie routing (check_decisions) outweigh the aggregate bar
        check_round(gpu, orc, synth.ARCH_SPLIT_CNN, grad=False)
        idx, counts = orc.sample()
        g = gpu.cut(pkg.binding.GCPSL_CUT_GRAD).reshape(2, B, -1).astype(np.float64)
        o = orc.cut(1).reshape(2, B, -1)
        for n in range(2):
            own = ds.owner[idx[n]]
            act = np.count_nonzero(counts[n])
            scale = B / (act * counts[n][own])
            assert rel_l2(g[n] / scale[:, None], o[n] / scale[:, None]) < REL_L2, (t, n)
            assert rel_l2(g[n], o[n]) < 0.1, (t, n)   # the factors themselves agree
    assert (orc.stats()[1] == 0).any()          # a cluster waited in the last round


def test_ragged_batch_nesterov_wd_label_smoothing():
    """B = 24 (not a power of two), C = 6, Nesterov, weight decay, label
    smoothing."""
    ds, assign, params = _splitcnn_small(C=6, n=6144, K=36, seed=5)
    kw = dict(lr=0.03, momentum=0.9, weight_decay=5e-4, nesterov=True, label_smoothing=0.1)
    gpu, orc = pair(synth.ARCH_SPLIT_CNN, 36, 6, assign, 24, 0, ds, params, True, **kw)
    for _ in range(3):
        check_round(gpu, orc, synth.ARCH_SPLIT_CNN)


def test_batch_of_one():
    """Degenerate batch: B = 1 (one client supplies the only example)."""
    ds, assign, params = _splitcnn_small(n=512, K=8)
    gpu, orc = pair(synth.ARCH_SPLIT_CNN, 8, 2, assign, 1, 1, ds, params, True, momentum=0.9)
    for _ in range(3):
        check_round(gpu, orc, synth.ARCH_SPLIT_CNN, grad=False)
    _, counts = gpu.sample()
    assert (counts.sum(1) == 1).all()


def test_largest_batch():
    """B = 1024, the largest batch gcpsl_init accepts (one sampler block of
    1024 threads per cluster), two clusters: one round against the oracle,
    and B = 1025 rejected."""
    ds, assign, params = _splitcnn_small(C=2, n=4096, K=16, seed=9)
    gpu, orc = pair(synth.ARCH_SPLIT_CNN, 16, 2, assign, 1024, 0, ds, params, True,
                    momentum=0.9)
    check_round(gpu, orc, synth.ARCH_SPLIT_CNN)
    _, counts = gpu.sample()
    assert (counts.sum(1) == 1024).all()
    gpu.close()
    with pytest.raises(pkg.binding.GcpslError):
        pkg.Context(synth.ARCH_SPLIT_CNN, 16, 1, np.zeros(16, np.int32), 1025, 0, 4, ds.images,
                    ds.labels, ds.owner, params)


def test_grouped_equals_serialized_bit_exact():
    """C clusters in one context == C one-cluster contexts (cluster_id_base=n):
    bit-identical parameters, momentum, cuts and samples."""
    ds, assign, params = _splitcnn_small(C=3, n=3072, K=24)
    kw = dict(lr=0.05, momentum=0.9)
    grouped = pkg.Context(1, 24, 3, assign, 32, 0, 4, ds.images, ds.labels, ds.owner, params,
                          bf16=True, **kw)
    alone = [pkg.Context(1, 24, 1, np.where(assign == n, 0, -1).astype(np.int32), 32, 0, 4,
                         ds.images, ds.labels, ds.owner, params, bf16=True, cluster_id_base=n,
                         **kw) for n in range(3)]
    for _ in range(3):
        grouped.step()
        for a in alone:
            a.step()
    gi, _ = grouped.sample()
    gz = grouped.cut(pkg.binding.GCPSL_CUT_GRAD)
    for n, a in enumerate(alone):
        ai, _ = a.sample()
        assert (ai[0] == gi[n]).all()
        assert (a.all_params(0) == grouped.all_params(n)).all()
        assert (a.momentum(0) == grouped.momentum(n)).all()
        assert (a.cut(pkg.binding.GCPSL_CUT_GRAD)[0] == gz[n]).all()


def test_data_on_host_is_identical():
    ds, assign, params = _splitcnn_small()
    a = pkg.Context(1, 32, 2, assign, 32, 2, 4, ds.images, ds.labels, ds.owner, params, bf16=True,
                    momentum=0.9)
    b = pkg.Context(1, 32, 2, assign, 32, 2, 4, ds.images, ds.labels, ds.owner, params, bf16=True,
                    momentum=0.9, data_on_host=True)
    for _ in range(3):
        la, _ = a.step(stats=True)
        lb, _ = b.step(stats=True)
        assert (la == lb).all()
    assert (a.all_params(1) == b.all_params(1)).all()


def test_rerun_is_deterministic():
    ds, assign, params = _splitcnn_small()
    runs = []
    for _ in range(2):
        g = pkg.Context(1, 32, 2, assign, 32, 2, 4, ds.images, ds.labels, ds.owner, params,
                        bf16=True, momentum=0.9)
        for _ in range(3):
            g.step()
        runs.append((g.all_params(0), g.cut(1)))
        g.close()
    assert (runs[0][0] == runs[1][0]).all() and (runs[0][1] == runs[1][1]).all()


def test_graph_replay_equals_eager_bit_exact():
    """Rounds replayed from CUDA graphs (timed and untimed copies, across an
    epoch boundary and fusions) equal eagerly launched rounds bit for bit."""
    ds, assign, params = _splitcnn_small(C=2, n=640, K=16)
    runs = []
    for graph in (False, True):
        g = pkg.Context(1, 16, 2, assign, 32, 4, 4, ds.images, ds.labels, ds.owner, params,
                        bf16=True, momentum=0.9)
        g.set_graph(graph)
        losses = []
        for t in range(11):
            g.set_timing(t % 3 == 1)        # alternate timed / untimed variants
            losses.append(g.step(stats=True)[0])
        kt = g.kernel_times()
        runs.append((np.stack([g.all_params(n) for n in range(2)]),
                     np.stack([g.momentum(n) for n in range(2)]), g.cut(1), np.array(losses)))
        g.close()
        assert sum(n for n, _ in kt.values()) > 0
    for a, b in zip(runs[0], runs[1]):
        assert (a == b).all()


def test_fusion_matches_eq5():
    """Explicit fusion of diverged replicas: Eq. 5 with the context's q."""
    ds, assign, params = _splitcnn_small(C=4, n=4096, K=32)
    gpu = pkg.Context(1, 32, 4, assign, 32, 0, 4, ds.images, ds.labels, ds.owner, params,
                      bf16=True, momentum=0.9)
    for _ in range(2):
        gpu.step()
    before = np.stack([gpu.all_params(n) for n in range(4)])
    mom_before = np.stack([gpu.momentum(n) for n in range(4)])
    sizes = configs.cluster_sizes(ds.owner, assign, 4)
    q = sizes / sizes.sum()
    expect = oracle.fuse_arrays(q, before)
    gpu.fuse()
    for n in range(4):
        got = gpu.all_params(n)
        assert rel_l2(got, expect) < FUSE_REL
        assert np.abs(got - expect).max() <= 4e-7 * np.abs(expect).max()
        assert (gpu.momentum(n) == mom_before[n]).all()     # optimiser state not fused
    gpu.fuse()                                              # identical replicas: identity
    assert (gpu.all_params(2) == got).all()


def test_splitcnn_c4_full_size():
    """The 50,000-image, K=256, C=4, B=64 workload in the benchmarked launch
    configuration: the first round of all four clusters against the oracle,
    and every cluster's sample against the oracle's sampler functions."""
    w = configs.WORKLOADS["splitcnn_c4"]
    ds, assign, params = configs.build_inputs(w)
    gpu, orc = pair(w.arch, w.num_clients, w.num_clusters, assign, w.B, w.F, ds, params, True,
                    lr=w.lr, momentum=w.momentum)
    check_round(gpu, orc, w.arch)
    gi, gc = gpu.sample()
    _, active = gpu.step(stats=True)   # round 2 from the GPU's own state: sampler only
    gi, gc = gpu.sample()
    assert (gc.sum(1) == w.B).all()
    for m in range(w.num_clusters):
        ids = np.flatnonzero(assign[ds.owner] == m).astype(np.int32)
        perm = oracle.epoch_perm(ids, m, 0, 4)
        idx, counts, act = oracle.sample_round(perm, 1, w.B, ds.owner, w.num_clients)
        assert (gi[m] == idx).all() and (gc[m] == counts).all() and active[m] == act


def _first_round_per_cluster(name, clusters):
    """A full-size workload in the benchmarked launch configuration: the
    GPU takes its first round with every cluster; selected clusters are
    re-run alone by the oracle (a one-cluster context with the same cluster
    id, so the same Philox stream) and compared slice by slice."""
    w = configs.WORKLOADS[name]
    ds, assign, params = configs.build_inputs(w)
    gpu = pkg.Context(w.arch, w.num_clients, w.num_clusters, assign, w.B, w.F, 4, ds.images,
                      ds.labels, ds.owner, params, lr=w.lr, momentum=w.momentum, bf16=True)
    loss, active = gpu.step(stats=True)
    gi, gc = gpu.sample()
    assert (gc.sum(1) == w.B).all()
    cut_act = gpu.cut(pkg.binding.GCPSL_CUT_ACT)
    cut_grad = gpu.cut(pkg.binding.GCPSL_CUT_GRAD)
    for m in clusters:
        sub = np.where(assign == m, 0, -1).astype(np.int32)
        orc = oracle.Oracle(w.arch, w.num_clients, 1, sub, w.B, w.F, 4, ds.images, ds.labels,
                            ds.owner, params, lr=w.lr, momentum=w.momentum, bf16=True,
                            cluster_base=m)
        orc.set_tie_tol(DECISION_TOL[True])
        orc.step()
        oi, oc = orc.sample()
        assert (gi[m] == oi[0]).all() and (gc[m] == oc[0]).all(), f"cluster {m}: sample"
        ol, oa = orc.stats()
        assert active[m] == oa[0]
        assert abs(loss[m] - ol[0]) < LOSS_ABS, (m, loss[m], ol[0])
        assert rel_l2(cut_act[m], orc.cut(0).reshape(cut_act[m].shape)) < REL_L2
        assert check_decisions(gpu, orc, w.arch, gpu_clusters=[m]) > 0.9
        assert rel_l2(cut_grad[m], orc.cut(1).reshape(cut_grad[m].shape)) < REL_L2
        gp, op = gpu.all_params(m), orc.all_params(0)
        assert rel_l2(gp, op) < REL_L2, ("params", m)
        assert rel_l2(gp - params, op - params) < REL_L2, ("update", m)
        del orc
    gpu.close()


def test_splitcnn_c16_full_size_sampled_clusters():
    """C=16 size-balanced clusters (50,000 images, K=256, B=64)."""
    _first_round_per_cluster("splitcnn_c16", [0, 7, 15])


def test_splitcnn_c64_full_size_sampled_clusters():
    """C=64 label-aware clusters (50,000 images, K=256, B=64): many small
    replica GEMMs in one grouped launch."""
    _first_round_per_cluster("splitcnn_c64", [0, 21, 42, 63])
