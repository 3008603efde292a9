"""Pins of the CPU oracle against facts fixed outside it.

Each test ties one part of the oracle to something other than itself:
published known-answer vectors (Philox), the invariants of Eq. 1-3, brute
force, closed forms, finite differences, and PyTorch's own fp64 conv /
max-pool / cross-entropy / SGD routines (which the oracle does not call).
"""
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

import oracle
from paper_2609_29395_gb300 import synth, clustering

GOLD = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------
# Philox4x32-10
# --------------------------------------------------------------------------
def _kat_rows():
    rows = []
    for line in open(os.path.join(GOLD, "philox4x32_10_kat.txt")):
        if line.startswith("#") or not line.strip():
            continue
        v = [int(t, 16) for t in line.split()]
        rows.append((v[:4], v[4:6], v[6:10]))
    return rows


@pytest.mark.parametrize("ctr,key,expect", _kat_rows())
def test_philox_known_answers(ctr, key, expect):
    assert list(oracle.philox4x32_10(ctr, key)) == expect


# --------------------------------------------------------------------------
# Sampler (Eq. 1, epoch rule of Section III-A, Eq. 3)
# --------------------------------------------------------------------------
def _keys(ids, cluster, epoch, seed):
    key = [seed & 0xFFFFFFFF, seed >> 32]
    k64 = []
    for j in ids:
        o = oracle.philox4x32_10([int(j), epoch, cluster, 0], key)
        k64.append((int(o[0]) << 32) | int(o[1]))
    return k64


def test_epoch_perm_is_the_key_order():
    rng = np.random.default_rng(11)
    ids = np.sort(rng.choice(5000, size=300, replace=False)).astype(np.int32)
    seed = 0x1234_5678_9ABC_DEF0
    perm = oracle.epoch_perm(ids, 3, 7, seed)
    k = _keys(ids, 3, 7, seed)
    expect = [j for _, j in sorted(zip(k, ids.tolist()))]
    assert perm.tolist() == expect
    # a different epoch or cluster gives a different order
    assert oracle.epoch_perm(ids, 3, 8, seed).tolist() != expect
    assert oracle.epoch_perm(ids, 4, 7, seed).tolist() != expect


def test_epoch_perm_uniform_chi2():
    """Position of each id over many epochs is uniform (chi-square)."""
    from scipy.stats import chisquare
    ids = np.arange(6, dtype=np.int32) * 5 + 1
    E = 3000
    pos = np.zeros((6, 6))
    for e in range(E):
        p = oracle.epoch_perm(ids, 0, e, 4)
        for i, j in enumerate(p):
            pos[(j - 1) // 5, i] += 1
    stat, pval = chisquare(pos.ravel(), np.full(36, E / 6))
    assert pval > 1e-4, (stat, pval)


def _small_world(seed=5, n=600, K=24, C=3):
    rng = np.random.default_rng(seed)
    owner = rng.integers(0, K, size=n).astype(np.int32)
    assign = clustering.random_clustering(K, C, seed)
    return owner, assign


def test_sample_round_invariants():
    owner, assign = _small_world()
    K, C, B = 24, 3, 16
    for n in range(C):
        ids = np.flatnonzero(assign[owner] == n).astype(np.int32)
        holdings = np.bincount(owner[ids], minlength=K)
        members = np.flatnonzero(assign == n)
        r = ids.size // B
        perm = oracle.epoch_perm(ids, n, 0, 4)
        assert sorted(perm.tolist()) == ids.tolist()
        seen = []
        cum = np.zeros(K, dtype=np.int64)
        for s in range(r):
            idx, counts, act = oracle.sample_round(perm, s, B, owner, K)
            assert counts.sum() == B                                   # Eq. 1
            assert (counts <= holdings).all()
            assert (counts[np.setdiff1d(np.arange(K), members)] == 0).all()
            assert act == (counts > 0).sum() <= min(B, members.size)   # |A| <= B
            rho = 1 - act / members.size
            assert rho >= max(0.0, 1 - B / members.size) - 1e-12       # Eq. 3
            key = list(zip(owner[idx].tolist(), idx.tolist()))
            assert key == sorted(key)
            assert (np.bincount(owner[idx], minlength=K) == counts).all()
            cum += counts
            seen += idx.tolist()
        assert (cum <= holdings).all()
        assert len(seen) == len(set(seen)) == r * B                     # once per epoch


def test_gpsl_bound_worked_values():
    for line in open(os.path.join(GOLD, "gpsl_bounds.txt")):
        if line.startswith("#") or not line.strip():
            continue
        K, B, bound = line.split()
        assert max(0.0, 1 - int(B) / int(K)) == pytest.approx(float(bound))


# --------------------------------------------------------------------------
# Forward / backward
# --------------------------------------------------------------------------
def _torch_model(arch, blob):
    """fp64 PyTorch forward of the split model from a canonical blob."""
    spec = synth.ARCHS[arch]
    convs = spec["client"] + spec["server"]
    t = torch.from_numpy(np.asarray(blob, dtype=np.float64)).clone().requires_grad_(True)
    off = 0
    ws = []
    for (cin, cout, _h, _w, pool) in convs:
        nw = cout * cin * 9
        ws.append((t[off:off + nw].view(cout, cin, 3, 3), t[off + nw:off + nw + cout], pool))
        off += nw + cout
    fin, fout = spec["fc"]
    fw = t[off:off + fin * fout].view(fout, fin)
    fb = t[off + fin * fout:off + fin * fout + fout]
    ncl = len(spec["client"])

    def fwd(x):
        z = None
        for i, (w, b, pool) in enumerate(ws):
            x = Fn.relu(Fn.conv2d(x, w, b, padding=1))
            if pool:
                x = Fn.max_pool2d(x, 2)
            if i == ncl - 1:
                z = x
                z.retain_grad()
        return Fn.linear(x.flatten(1), fw, fb), z
    return t, fwd


@pytest.mark.parametrize("arch,B", [(synth.ARCH_TINY_CNN, 4), (synth.ARCH_SPLIT_CNN, 2)])
def test_forward_backward_matches_torch_fp64(arch, B):
    rng = np.random.default_rng(3)
    blob = synth.init_params(arch, seed=9).astype(np.float64)
    x = rng.standard_normal((B, 3, 32, 32))
    y = rng.integers(0, 10, size=B).astype(np.int32)
    loss, grad, ca, cg, logits = oracle.forward_backward(arch, blob, x, y)
    t, fwd = _torch_model(arch, blob)
    out, z = fwd(torch.from_numpy(x))
    tl = Fn.cross_entropy(out, torch.from_numpy(y.astype(np.int64)))
    tl.backward()
    assert loss == pytest.approx(tl.item(), rel=1e-12, abs=1e-12)
    np.testing.assert_allclose(logits, out.detach().numpy(), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(grad, t.grad.numpy(), rtol=1e-9, atol=1e-13)
    np.testing.assert_allclose(ca, z.detach().numpy().ravel(), rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(cg, z.grad.numpy().ravel(), rtol=1e-9, atol=1e-14)


def test_label_smoothing_matches_torch():
    arch, B = synth.ARCH_TINY_CNN, 3
    rng = np.random.default_rng(4)
    blob = synth.init_params(arch, seed=2).astype(np.float64)
    x = rng.standard_normal((B, 3, 32, 32))
    y = rng.integers(0, 10, size=B).astype(np.int32)
    loss, grad, *_ = oracle.forward_backward(arch, blob, x, y, label_smoothing=0.1)
    t, fwd = _torch_model(arch, blob)
    out, _ = fwd(torch.from_numpy(x))
    tl = Fn.cross_entropy(out, torch.from_numpy(y.astype(np.int64)), label_smoothing=0.1)
    tl.backward()
    assert loss == pytest.approx(tl.item(), rel=1e-12)
    np.testing.assert_allclose(grad, t.grad.numpy(), rtol=1e-9, atol=1e-13)


def test_finite_differences():
    """Central differences of the oracle's own loss agree with its gradient."""
    arch, B = synth.ARCH_TINY_CNN, 2
    rng = np.random.default_rng(8)
    blob = synth.init_params(arch, seed=5).astype(np.float64)
    x = rng.standard_normal((B, 3, 32, 32))
    y = np.array([3, 7], dtype=np.int32)
    _, grad, *_ = oracle.forward_backward(arch, blob, x, y)
    # a few coordinates from every tensor (conv0 w/b, conv1 w/b, fc w/b)
    bounds = np.cumsum([0, 432, 16, 4608, 32, 20480, 10])
    picks = [int(rng.integers(bounds[i], bounds[i + 1])) for i in range(6) for _ in range(4)]
    h = 1e-6
    for p in picks:
        bp, bm = blob.copy(), blob.copy()
        bp[p] += h
        bm[p] -= h
        lp = oracle.forward_backward(arch, bp, x, y, want_grad=False)[0]
        lm = oracle.forward_backward(arch, bm, x, y, want_grad=False)[0]
        fd = (lp - lm) / (2 * h)
        assert fd == pytest.approx(grad[p], rel=1e-5, abs=1e-9), p


def test_zero_weights_give_ln10():
    for arch in (synth.ARCH_TINY_CNN, synth.ARCH_SPLIT_CNN):
        P = oracle.num_params(arch, 0) + oracle.num_params(arch, 1)
        x = np.random.default_rng(0).standard_normal((2, 3, 32, 32))
        loss, *_ = oracle.forward_backward(arch, np.zeros(P), x, np.array([1, 9], np.int32),
                                           want_grad=False)
        assert loss == pytest.approx(math.log(10.0), rel=1e-15)


def test_bf16_mode_rounds_only():
    """bf16 operand mode stays close to fp64 (a rounding mode, not a new op)."""
    arch, B = synth.ARCH_TINY_CNN, 4
    rng = np.random.default_rng(1)
    blob = synth.init_params(arch, seed=1).astype(np.float64)
    x = rng.standard_normal((B, 3, 32, 32))
    y = rng.integers(0, 10, size=B).astype(np.int32)
    l64, g64, *_ = oracle.forward_backward(arch, blob, x, y)
    l16, g16, *_ = oracle.forward_backward(arch, blob, x, y, bf16=True)
    assert abs(l64 - l16) < 2e-2
    assert np.linalg.norm(g16 - g64) / np.linalg.norm(g64) < 5e-2
    assert l64 != l16


# --------------------------------------------------------------------------
# Fusion (Eq. 5)
# --------------------------------------------------------------------------
def test_fusion_identity():
    rng = np.random.default_rng(2)
    th = rng.standard_normal(1000).astype(np.float32).astype(np.float64)
    q = np.array([0.1, 0.2, 0.3, 0.4])
    out = oracle.fuse_arrays(q, np.stack([th] * 4))
    np.testing.assert_allclose(out, th, rtol=1e-15)
    assert (out.astype(np.float32) == th.astype(np.float32)).all()


def test_fusion_closed_form():
    C, P = 5, 64
    q = np.arange(1, C + 1, dtype=np.float64)
    q /= q.sum()
    theta = np.stack([np.full(P, float(n)) for n in range(C)])
    out = oracle.fuse_arrays(q, theta)
    np.testing.assert_allclose(out, np.full(P, sum(q[n] * n for n in range(C))), rtol=1e-15)


# --------------------------------------------------------------------------
# Whole rounds: C = 1 is GPSL; concurrent == sequential; fusion in the loop
# --------------------------------------------------------------------------
def _tiny_world(n=256, K=8, seed=0):
    ds = synth.make_dataset(n, 10, K, 0.5, balanced=False, seed_data=seed, seed_split=seed + 1)
    return ds


def test_single_cluster_is_gpsl_against_torch_sgd():
    """C=1 with every client in it is plain GPSL: replay its batches through
    PyTorch fp64 autograd and torch.optim.SGD(momentum=0.9)."""
    arch, B, K = synth.ARCH_TINY_CNN, 8, 8
    ds = _tiny_world(K=K)
    blob = synth.init_params(arch, seed=3)
    orc = oracle.Oracle(arch, K, 1, np.zeros(K, np.int32), B, 0, 4, ds.images, ds.labels,
                        ds.owner, blob, lr=0.05, momentum=0.9)
    t, fwd = _torch_model(arch, blob.astype(np.float64))
    opt = torch.optim.SGD([t], lr=0.05, momentum=0.9)
    for _ in range(4):
        orc.step()
        idx, counts = orc.sample()
        assert counts.sum() == B
        opt.zero_grad()
        out, _ = fwd(torch.from_numpy(ds.images[idx[0]].astype(np.float64)))
        Fn.cross_entropy(out, torch.from_numpy(ds.labels[idx[0]].astype(np.int64))).backward()
        opt.step()
        np.testing.assert_allclose(orc.all_params(0), t.detach().numpy(), rtol=1e-10, atol=1e-12)


def test_concurrent_equals_sequential_then_fusion():
    """C clusters in one context == each cluster alone (cluster_base = n),
    and the context's fusion == Eq. 5 over the separate replicas."""
    arch, B, K, C = synth.ARCH_TINY_CNN, 8, 8, 2
    ds = _tiny_world(K=K, seed=2)
    assign = clustering.random_clustering(K, C, 2)
    blob = synth.init_params(arch, seed=3)
    common = dict(lr=0.05, momentum=0.9)
    grouped = oracle.Oracle(arch, K, C, assign, B, 0, 4, ds.images, ds.labels, ds.owner, blob,
                            **common)
    alone = [oracle.Oracle(arch, K, 1, np.where(assign == n, 0, -1).astype(np.int32), B, 0, 4,
                           ds.images, ds.labels, ds.owner, blob, cluster_base=n, **common)
             for n in range(C)]
    for _ in range(3):
        grouped.step()
        for a in alone:
            a.step()
    gi, gc = grouped.sample()
    for n in range(C):
        ai, ac = alone[n].sample()
        assert (ai[0] == gi[n]).all() and (ac[0] == gc[n]).all()
        assert (alone[n].all_params(0) == grouped.all_params(n)).all()
    q = grouped.q()
    sizes = np.bincount(assign[ds.owner], minlength=C)
    np.testing.assert_allclose(q, sizes / sizes.sum(), rtol=0, atol=0)
    fused = oracle.fuse_arrays(q, np.stack([a.all_params(0) for a in alone]))
    grouped.fuse()
    for n in range(C):
        assert (grouped.all_params(n) == fused).all()


def test_fusion_every_F_rounds_in_the_loop():
    arch, B, K, C, F = synth.ARCH_TINY_CNN, 8, 8, 2, 2
    ds = _tiny_world(K=K, seed=3)
    assign = clustering.random_clustering(K, C, 1)
    blob = synth.init_params(arch, seed=3)
    orc = oracle.Oracle(arch, K, C, assign, B, F, 4, ds.images, ds.labels, ds.owner, blob,
                        lr=0.05)
    orc.step()
    assert not (orc.all_params(0) == orc.all_params(1)).all()
    orc.step()                                   # round 2: fused, replicas equal
    assert (orc.all_params(0) == orc.all_params(1)).all()


def test_init_rejects_bad_inputs():
    arch, K = synth.ARCH_TINY_CNN, 8
    ds = _tiny_world(K=K)
    blob = synth.init_params(arch)
    with pytest.raises(ValueError):   # cluster smaller than B
        oracle.Oracle(arch, K, 1, np.zeros(K, np.int32), 10_000, 0, 4, ds.images, ds.labels,
                      ds.owner, blob)
    with pytest.raises(ValueError):   # assignment out of range
        oracle.Oracle(arch, K, 2, np.full(K, 2, np.int32), 8, 0, 4, ds.images, ds.labels,
                      ds.owner, blob)


# --------------------------------------------------------------------------
# Training augmentation (Section V-A: random crop + horizontal flip)
# --------------------------------------------------------------------------
def test_augment_image_is_padded_crop_then_flip():
    """The oracle's augmentation equals numpy's zero-pad by 4, crop at
    (dy, dx), then left-right mirror, for every offset and both flips."""
    rng = np.random.default_rng(3)
    img = rng.normal(size=(3, 32, 32)).astype(np.float32)
    padded = np.pad(img.astype(np.float64), ((0, 0), (4, 4), (4, 4)))
    for dy in range(9):
        for dx in range(9):
            for flip in (0, 1):
                ref = padded[:, dy:dy + 32, dx:dx + 32]
                if flip:
                    ref = ref[:, :, ::-1]
                got = oracle.augment_image(img, dy, dx, flip)
                assert np.array_equal(got, ref), (dy, dx, flip)


def test_augment_params_range_uniformity_and_stream():
    """Offsets in [0, 8], flips in {0, 1}, each close to uniform (chi^2 over
    many draws); draws differ between rounds, clusters and positions, and
    equal the Philox definition (counter (pos, t, cluster, 1), key = seed)."""
    seed = 0x1234ABCD5678
    n = 9 * 800
    draws = np.array([oracle.augment_params(seed, t, c, p)
                      for t in range(20) for c in range(4) for p in range(n // 80)])
    assert draws.shape[0] == n
    assert draws[:, :2].min() == 0 and draws[:, :2].max() == 8
    assert set(np.unique(draws[:, 2])) == {0, 1}
    for col in (0, 1):
        cnt = np.bincount(draws[:, col], minlength=9)
        chi2 = ((cnt - n / 9) ** 2 / (n / 9)).sum()
        assert chi2 < 30.0, (col, cnt)            # 8 dof: p(chi2 > 30) < 3e-4
    assert abs(draws[:, 2].mean() - 0.5) < 0.03
    o = [int(v) for v in oracle.philox4x32_10([5, 7, 3, 1], [seed & 0xFFFFFFFF, seed >> 32])]
    assert oracle.augment_params(seed, 7, 3, 5) == ((o[0] * 9) >> 32, (o[1] * 9) >> 32, o[2] & 1)


def test_oracle_round_uses_the_augmented_batch():
    """With augmentation, a round's loss equals the forward pass on the
    sampled images augmented with that round's draws (and differs from the
    plain batch)."""
    ds = synth.make_dataset(256, 10, 8, 0.5, balanced=False, seed_data=1, seed_split=2)
    assign = clustering.random_clustering(8, 2, 3)
    arch = synth.ARCH_TINY_CNN
    params = synth.init_params(arch, seed=4).astype(np.float64)
    B, seed = 16, 9
    for aug in (True, False):
        orc = oracle.Oracle(arch, 8, 2, assign, B, 0, seed, ds.images, ds.labels, ds.owner,
                            params, augment=aug)
        orc.step()
        idx, _ = orc.sample()
        loss, _ = orc.stats()
        for m in range(2):
            x = ds.images[idx[m]].astype(np.float64)
            if aug:
                x = np.stack([oracle.augment_image(ds.images[i], *oracle.augment_params(seed, 0, m, b))
                              for b, i in enumerate(idx[m])])
            ref = oracle.forward_backward(arch, params, x, ds.labels[idx[m]])[0]
            assert abs(ref - loss[m]) < 1e-12 * max(1.0, abs(ref))


# --------------------------------------------------------------------------
# Epoch schedule with the fusion barrier (Section IV-C, Eq. 6)
# --------------------------------------------------------------------------
def test_epoch_schedule_barrier_and_fusion():
    """F = -1: cluster n takes r_n = n_c / B local rounds per system epoch of
    R = max r_n rounds, then waits (parameters, momentum and sample frozen,
    loss and |A| reported 0); after R rounds the replicas are fused with q
    (Eq. 5).  Its first min r_n rounds equal the lockstep schedule's."""
    ds = synth.make_dataset(600, 10, 12, 0.5, balanced=False, seed_data=5, seed_split=6)
    rng = np.random.default_rng(7)
    assign = rng.choice(3, size=12, p=[0.55, 0.3, 0.15]).astype(np.int32)
    assign[:3] = [0, 1, 2]
    arch = synth.ARCH_TINY_CNN
    params = synth.init_params(arch, seed=8)
    B = 16
    sizes = np.bincount(assign[ds.owner], minlength=3)
    r = clustering.schedule_rounds(sizes, B)
    R = int(r.max())
    assert len(set(r.tolist())) > 1, r          # unequal epochs
    kw = dict(lr=0.05, momentum=0.9)
    ep = oracle.Oracle(arch, 12, 3, assign, B, -1, 4, ds.images, ds.labels, ds.owner, params, **kw)
    ls = oracle.Oracle(arch, 12, 3, assign, B, 0, 4, ds.images, ds.labels, ds.owner, params, **kw)
    seen = [set() for _ in range(3)]
    for t in range(R):
        before = [ep.all_params(n) for n in range(3)]
        ep.step()
        ls.step()
        idx, counts = ep.sample()
        loss, active = ep.stats()
        last = t == R - 1
        for n in range(3):
            if t < r[n]:
                assert loss[n] > 0 and active[n] > 0
                seen[n].update(idx[n].tolist())
                if t < r.min():
                    li, _ = ls.sample()
                    assert (idx[n] == li[n]).all()
                if not last:
                    assert not np.array_equal(ep.all_params(n), before[n])
            else:
                assert loss[n] == 0 and active[n] == 0
                if not last:
                    assert np.array_equal(ep.all_params(n), before[n])
        if t == R - 2:
            pre_fuse = [ep.all_params(n) for n in range(3)]
    for n in range(3):
        assert len(seen[n]) == r[n] * B                 # each example at most once
    q = ep.q()
    fused = ep.all_params(0)
    for n in range(3):
        assert np.array_equal(ep.all_params(n), fused)
    # every cluster but the longest waited in round R - 1 (its parameters
    # before the fusion are those after round R - 2); the longest one's
    # trajectory is the lockstep run's (same batches, no fusion yet)
    longest = int(np.argmax(r))
    assert sorted(r.tolist()).count(R) == 1
    expect = sum(q[n] * pre_fuse[n] for n in range(3) if n != longest) + \
        q[longest] * ls.all_params(longest)
    np.testing.assert_allclose(fused, expect, rtol=0, atol=1e-12 * np.abs(expect).max())
    s, e = clustering.ideal_schedule_speedup(sizes, B)
    assert abs(s - r.sum() / R) < 1e-12 and abs(e - s / 3) < 1e-12


@pytest.mark.parametrize("arch", [synth.ARCH_TINY_CNN, synth.ARCH_SPLIT_CNN])
def test_client_average_is_the_mean_of_per_client_gradients(arch):
    """client_average (Sec. IV-B's other reading): the client segment's
    gradient is the unweighted mean over the round's active clients of each
    client's mean-loss gradient, each computed by an independent forward /
    backward of that client's examples alone; the server segment keeps the
    gradient of the batch-mean loss.  fp64, lr 1, no momentum: the update
    is minus the gradient."""
    B, K = 16, 8
    ds = _tiny_world(K=K, seed=4)
    blob = synth.init_params(arch, seed=5).astype(np.float64)
    orc = oracle.Oracle(arch, K, 1, np.zeros(K, np.int32), B, 0, 4, ds.images, ds.labels,
                        ds.owner, blob, lr=1.0, client_average=True)
    orc.step()
    idx, counts = orc.sample()
    idx = idx[0]
    owners = ds.owner[idx]
    active = np.flatnonzero(counts[0])
    assert len(active) > 1 and len(set(counts[0][active])) > 1   # unequal b_k
    g = blob - orc.all_params(0)
    pc = oracle.num_params(arch, 0)
    want_c = np.zeros(pc)
    for k in active:
        sel = idx[owners == k]
        gk = oracle.forward_backward(arch, blob, ds.images[sel].astype(np.float64),
                                     ds.labels[sel])[1]
        want_c += gk[:pc] / len(active)
    full = oracle.forward_backward(arch, blob, ds.images[idx].astype(np.float64),
                                   ds.labels[idx])[1]
    np.testing.assert_allclose(g[:pc], want_c, rtol=0, atol=1e-10 * np.abs(want_c).max())
    np.testing.assert_allclose(g[pc:], full[pc:], rtol=0, atol=1e-10 * np.abs(full[pc:]).max())
    # and it differs from the example-weighted default when the b_k differ
    assert np.abs(g[:pc] - full[:pc]).max() > 1e-3 * np.abs(full[:pc]).max()
