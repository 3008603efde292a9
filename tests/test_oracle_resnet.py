"""Pins of the oracle's ResNet-18 split (architectures 2 and 3, 10- and
100-way heads) against PyTorch's
fp64 autograd, written here from the module definitions (conv2d,
group_norm, batch_norm in training mode, relu, avg_pool2d, linear,
cross_entropy) -- none of the oracle's code.  CPU only."""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from paper_2609_29395_gb300 import synth

RES = synth.ARCH_RESNET18
RES100 = synth.ARCH_RESNET18_C100


def torch_model(blob, x, y, bn_state, label_smoothing=0.0, arch=RES, groups=32, eps=1e-5,
                momentum=0.1):
    """Loss, parameter tensors (requires_grad), cut activation (retained
    grad), logits and the BatchNorm state after the batch, with the blob in
    PyTorch's named_parameters() order."""
    names = [n for n, _ in synth.param_shapes(arch, "client") + synth.param_shapes(arch, "server")]
    shapes = [s for _, s in synth.param_shapes(arch, "client") + synth.param_shapes(arch, "server")]
    prm, off = {}, 0
    for n, s in zip(names, shapes):
        k = int(np.prod(s))
        prm[n] = torch.tensor(blob[off:off + k].reshape(s), dtype=torch.float64,
                              requires_grad=True)
        off += k
    state = torch.tensor(bn_state, dtype=torch.float64)
    soff = [0]

    def bn(t, pre):
        c = t.shape[1]
        rm = state[soff[0]:soff[0] + c]
        rv = state[soff[0] + c:soff[0] + 2 * c]
        soff[0] += 2 * c
        return F.batch_norm(t, rm, rv, prm[pre + ".weight"], prm[pre + ".bias"], training=True,
                            momentum=momentum, eps=eps)

    def gn(t, pre):
        return F.group_norm(t, groups, prm[pre + ".weight"], prm[pre + ".bias"], eps=eps)

    h = F.relu(gn(F.conv2d(x, prm["conv1.weight"], padding=1), "bn1"))
    cut = None
    cin = 64
    for st, (width, stride) in enumerate(synth.RESNET_STAGES):
        norm = gn if st == 0 else bn
        for j in range(2):
            s = stride if j == 0 else 1
            pre = f"layer{st + 1}.{j}"
            o = F.relu(norm(F.conv2d(h, prm[pre + ".conv1.weight"], stride=s, padding=1),
                            pre + ".bn1"))
            o = norm(F.conv2d(o, prm[pre + ".conv2.weight"], padding=1), pre + ".bn2")
            if s != 1 or cin != width:
                sc = norm(F.conv2d(h, prm[pre + ".shortcut.0.weight"], stride=s),
                          pre + ".shortcut.1")
            else:
                sc = h
            h = F.relu(o + sc)
            cin = width
        if st == 0:
            cut = h
            cut.retain_grad()
    feat = F.avg_pool2d(h, 4).flatten(1)
    logits = F.linear(feat, prm["linear.weight"], prm["linear.bias"])
    loss = F.cross_entropy(logits, torch.tensor(y, dtype=torch.long),
                           label_smoothing=label_smoothing)
    return loss, [prm[n] for n in names], cut, logits, state.numpy()


def make_case(arch, labels):
    rng = np.random.default_rng(11)
    blob = synth.init_params(arch, seed=7).astype(np.float64)
    # non-trivial norm affine parameters
    off = 0
    for name, shape in synth.param_shapes(arch, "client") + synth.param_shapes(arch, "server"):
        k = int(np.prod(shape))
        if len(shape) == 1 and name != "linear.bias":
            blob[off:off + k] += rng.normal(0, 0.2, k)
        off += k
    B = len(labels)
    x = rng.normal(size=(B, 3, 32, 32))
    y = np.asarray(labels, dtype=np.int32)
    bn0 = oracle.initial_bn_state()
    bn0[:] += rng.uniform(0.0, 0.5, bn0.size)
    return blob, x, y, bn0


@pytest.fixture(scope="module")
def case():
    return make_case(RES, [3, 9, 0])


@pytest.fixture(scope="module")
def case100():
    # labels beyond the first ten rows of the head
    return make_case(RES100, [57, 3, 99])


def test_resnet_param_count_and_state_size():
    assert oracle.num_params(RES, 0) == synth.num_params(RES, "client") == 149824
    assert oracle.num_params(RES, 0) + oracle.num_params(RES, 1) == 11173962
    assert oracle.bn_state_size() == 8960
    st = oracle.initial_bn_state()
    assert set(np.unique(st)) == {0.0, 1.0} and st.sum() == 4480


@pytest.mark.parametrize("ls", [0.0, 0.1])
def test_resnet_matches_torch_fp64_autograd(case, ls):
    blob, x, y, bn0 = case
    loss, grad, ca, cg, logits, bn1 = oracle.resnet_forward_backward(
        blob, x, y, bn_state=bn0, label_smoothing=ls)
    tl, tparams, tcut, tlogits, tstate = torch_model(blob, torch.tensor(x), y, bn0, ls)
    tl.backward()
    tgrad = np.concatenate([p.grad.numpy().ravel() for p in tparams])
    assert abs(loss - tl.item()) < 1e-12 * max(1.0, abs(loss))
    np.testing.assert_allclose(logits, tlogits.detach().numpy(), rtol=0, atol=1e-11)
    np.testing.assert_allclose(ca, tcut.detach().numpy().ravel(), rtol=0, atol=1e-11)
    np.testing.assert_allclose(cg, tcut.grad.numpy().ravel(), rtol=0,
                               atol=1e-12 * np.abs(cg).max())
    scale = np.abs(tgrad).max()
    np.testing.assert_allclose(grad, tgrad, rtol=0, atol=1e-10 * scale)
    np.testing.assert_allclose(bn1, tstate, rtol=0, atol=1e-12)


@pytest.mark.parametrize("groups,eps,momentum", [(8, 1e-3, 0.2), (1, 1e-4, 1.0)])
def test_resnet_norm_hyperparameters_match_torch(case, groups, eps, momentum):
    """Other GroupNorm group counts, norm eps and BatchNorm momentum (the
    model description's gn_groups / norm_eps / bn_momentum) against PyTorch's
    group_norm / batch_norm with the same values."""
    blob, x, y, bn0 = case
    loss, grad, ca, cg, logits, bn1 = oracle.resnet_forward_backward(
        blob, x, y, bn_state=bn0, gn_groups=groups, norm_eps=eps, bn_momentum=momentum)
    tl, tparams, tcut, tlogits, tstate = torch_model(blob, torch.tensor(x), y, bn0,
                                                     groups=groups, eps=eps, momentum=momentum)
    tl.backward()
    tgrad = np.concatenate([p.grad.numpy().ravel() for p in tparams])
    assert abs(loss - tl.item()) < 1e-12 * max(1.0, abs(loss))
    np.testing.assert_allclose(ca, tcut.detach().numpy().ravel(), rtol=0, atol=1e-11)
    np.testing.assert_allclose(grad, tgrad, rtol=0, atol=1e-10 * np.abs(tgrad).max())
    np.testing.assert_allclose(bn1, tstate, rtol=0, atol=1e-12)
    # the defaults come back after the call
    l_def = oracle.resnet_forward_backward(blob, x, y, bn_state=bn0, want_grad=False)[0]
    t_def = torch_model(blob, torch.tensor(x), y, bn0)[0].item()
    assert abs(l_def - t_def) < 1e-12 * max(1.0, abs(t_def))
    with pytest.raises(ValueError):
        oracle.resnet_forward_backward(blob, x, y, bn_state=bn0, gn_groups=3)


def test_resnet_cut_scale_matches_torch(case):
    """The per-client average's cut scaling on the ResNet split: the client
    segment's gradient is the backward of (cut gradient x s_b) through the
    client (PyTorch: autograd.grad with those grad_outputs); the server's
    gradient and the loss are unchanged."""
    blob, x, y, bn0 = case
    s = np.array([0.5, 2.0, 1.25])
    loss, grad, ca, cg, logits, bn1 = oracle.resnet_forward_backward(
        blob, x, y, bn_state=bn0, cut_scale=s)
    plain = oracle.resnet_forward_backward(blob, x, y, bn_state=bn0)
    tl, tparams, tcut, tlogits, tstate = torch_model(blob, torch.tensor(x), y, bn0)
    tl.backward(retain_graph=True)
    pc = oracle.num_params(RES, 0)
    ncl = len(synth.param_shapes(RES, "client"))
    client = tparams[:ncl]
    go = tcut.grad.clone() * torch.tensor(s).view(-1, 1, 1, 1)
    tc = torch.autograd.grad(tcut, client, grad_outputs=go)
    want_c = np.concatenate([t.numpy().ravel() for t in tc])
    assert abs(loss - plain[0]) == 0.0
    np.testing.assert_allclose(grad[:pc], want_c, rtol=0, atol=1e-10 * np.abs(want_c).max())
    np.testing.assert_array_equal(grad[pc:], plain[1][pc:])
    np.testing.assert_allclose(cg, go.numpy().ravel(), rtol=0, atol=1e-12 * np.abs(cg).max())


def test_resnet100_param_count():
    assert oracle.num_params(RES100, 0) == oracle.num_params(RES, 0) == 149824
    assert oracle.num_params(RES100, 1) == synth.num_params(RES100, "server") == \
        oracle.num_params(RES, 1) + 90 * 512 + 90


@pytest.mark.parametrize("ls", [0.0, 0.1])
def test_resnet100_matches_torch_fp64_autograd(case100, ls):
    """The 100-way head (architecture 3) against PyTorch's linear +
    cross_entropy with its 100 classes, label smoothing spread over all 100."""
    blob, x, y, bn0 = case100
    loss, grad, ca, cg, logits, bn1 = oracle.resnet_forward_backward(
        blob, x, y, bn_state=bn0, label_smoothing=ls, classes=100)
    tl, tparams, tcut, tlogits, tstate = torch_model(blob, torch.tensor(x), y, bn0, ls,
                                                     arch=RES100)
    tl.backward()
    tgrad = np.concatenate([p.grad.numpy().ravel() for p in tparams])
    assert logits.shape == (3, 100)
    assert abs(loss - tl.item()) < 1e-12 * max(1.0, abs(loss))
    np.testing.assert_allclose(logits, tlogits.detach().numpy(), rtol=0, atol=1e-11)
    np.testing.assert_allclose(cg, tcut.grad.numpy().ravel(), rtol=0,
                               atol=1e-12 * np.abs(cg).max())
    np.testing.assert_allclose(grad, tgrad, rtol=0, atol=1e-10 * np.abs(tgrad).max())
    np.testing.assert_allclose(bn1, tstate, rtol=0, atol=1e-12)


def test_resnet100_zero_head_closed_form(case100):
    """Zero head weights and bias: every logit 0, so the loss is ln 100 with
    or without label smoothing, the bias gradient is 1/100 - mean_b t_b (t
    the smoothed target), and the cut gradient vanishes."""
    blob, x, y, bn0 = case100
    z = blob.copy()
    off = oracle.num_params(RES100, 0) + oracle.num_params(RES100, 1) - 100 * 512 - 100
    z[off:] = 0.0
    for ls in (0.0, 0.1):
        l0, g, _ca, cg, logits, _ = oracle.resnet_forward_backward(
            z, x, y, bn_state=bn0, label_smoothing=ls, classes=100)
        assert abs(l0 - np.log(100.0)) < 1e-13     # a 100-term fp64 sum
        assert np.abs(logits).max() == 0.0
        assert np.abs(cg).max() == 0.0
        want_db = np.full(100, 1.0 / 100) - np.bincount(y, minlength=100) * (1.0 - ls) / len(y) \
            - ls / 100
        np.testing.assert_allclose(g[-100:], want_db, rtol=0, atol=1e-15)


def test_resnet100_rejects_labels_outside_the_head(case100):
    blob, x, y, bn0 = case100
    with pytest.raises(RuntimeError):
        oracle.resnet_forward_backward(blob[:oracle.num_params(RES, 0) + oracle.num_params(RES, 1)],
                                       x, y, bn_state=bn0, classes=10)


def test_resnet_finite_differences(case):
    """Central differences of the loss on a few parameters of each kind."""
    blob, x, y, bn0 = case
    _, grad, *_ = oracle.resnet_forward_backward(blob, x, y, bn_state=bn0)
    names = synth.param_shapes(RES, "client") + synth.param_shapes(RES, "server")
    offs, o = {}, 0
    for n, s in names:
        offs[n] = o
        o += int(np.prod(s))
    picks = [offs["conv1.weight"] + 5, offs["bn1.weight"] + 3, offs["layer1.1.conv2.weight"] + 77,
             offs["layer2.0.shortcut.0.weight"] + 9, offs["layer3.1.bn2.bias"] + 4,
             offs["layer4.0.conv1.weight"] + 1234, offs["linear.weight"] + 99]
    # a small step keeps every ReLU on its side for most parameters: the
    # loss is only piecewise smooth
    h = 1e-7
    for i in picks:
        p = blob.copy()
        p[i] += h
        lp = oracle.resnet_forward_backward(p, x, y, bn_state=bn0, want_grad=False)[0]
        p[i] -= 2 * h
        lm = oracle.resnet_forward_backward(p, x, y, bn_state=bn0, want_grad=False)[0]
        fd = (lp - lm) / (2 * h)
        assert abs(fd - grad[i]) < 1e-5 * max(1.0, abs(grad[i])) + 1e-8, (i, fd, grad[i])


def test_resnet_bf16_mode_rounds_only_stored_values(case):
    """bf16 operand mode stays within bf16 rounding of the exact pass, and a
    zero-weight head gives the closed-form loss ln 10."""
    blob, x, y, bn0 = case
    l64 = oracle.resnet_forward_backward(blob, x, y, bn_state=bn0, want_grad=False)[0]
    l16 = oracle.resnet_forward_backward(blob, x, y, bn_state=bn0, bf16=True,
                                         want_grad=False)[0]
    assert abs(l64 - l16) < 2e-2 * abs(l64)
    z = blob.copy()
    off = oracle.num_params(RES, 0) + oracle.num_params(RES, 1) - 10 * 512 - 10
    z[off:] = 0.0
    l0 = oracle.resnet_forward_backward(z, x, y, bn_state=bn0, want_grad=False)[0]
    assert abs(l0 - np.log(10.0)) < 1e-14


def test_resnet_context_step_concurrent_equals_sequential_and_fusion():
    """An oracle context with two ResNet-18 clusters: one round equals each
    cluster run alone (same cluster id) bit for bit, the update of a
    replica is SGD on PyTorch's gradient of its sampled batch, and fusion
    averages parameters and BatchNorm running statistics with q (Eq. 5)."""
    from paper_2609_29395_gb300 import clustering
    ds = synth.make_dataset(96, 10, 8, 0.5, balanced=False, seed_data=3, seed_split=4)
    assign = clustering.random_clustering(8, 2, 5)
    blob = synth.init_params(RES, seed=9)
    B, lr = 4, 0.05
    kw = dict(lr=lr, momentum=0.9)
    both = oracle.Oracle(RES, 8, 2, assign, B, 0, 4, ds.images, ds.labels, ds.owner, blob, **kw)
    both.step()
    idx, _ = both.sample()
    for m in range(2):
        sub = np.where(assign == m, 0, -1).astype(np.int32)
        one = oracle.Oracle(RES, 8, 1, sub, B, 0, 4, ds.images, ds.labels, ds.owner, blob,
                            cluster_base=m, **kw)
        one.step()
        assert (one.all_params(0) == both.all_params(m)).all()
        assert (one.bn_state(0) == both.bn_state(m)).all()
        # SGD on PyTorch's gradient of the same batch (first round: v = g)
        x = ds.images[idx[m]].astype(np.float64)
        y = ds.labels[idx[m]]
        tl, tparams, _, _, tstate = torch_model(blob.astype(np.float64), torch.tensor(x), y,
                                                oracle.initial_bn_state())
        tl.backward()
        tgrad = np.concatenate([p.grad.numpy().ravel() for p in tparams])
        expect = blob.astype(np.float64) - lr * tgrad
        np.testing.assert_allclose(both.all_params(m), expect, rtol=0,
                                   atol=1e-10 * np.abs(expect).max())
        np.testing.assert_allclose(both.bn_state(m), tstate, rtol=0, atol=1e-12)
    p = np.stack([both.all_params(m) for m in range(2)])
    s = np.stack([both.bn_state(m) for m in range(2)])
    q = both.q()
    both.fuse()
    for m in range(2):
        np.testing.assert_allclose(both.all_params(m), q[0] * p[0] + q[1] * p[1], rtol=0,
                                   atol=1e-15)
        np.testing.assert_allclose(both.bn_state(m), q[0] * s[0] + q[1] * s[1], rtol=0,
                                   atol=1e-15)
