"""Seeded synthetic inputs for the GCPSL training step.

This module only draws random inputs: images, labels, the per-client data
split and the initial split-model parameters.  It holds none of the method's
arithmetic (no sampling, no forward/backward, no update, no fusion), so that
both the CUDA library and the CPU oracle can take their inputs from it.

Stand-in for CIFAR-10 and CIFAR-100 (Section V-A; the datasets are not
available here): 32x32x3 images with N(0,1) pixels and 10 or 100 classes.  Two
client splits: a per-class Dirichlet(alpha) draw over all clients, and the
extended-Dirichlet protocol of Section V-A (each client holds two classes,
each class is spread over its holders by a Dirichlet(alpha) draw).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

IMG_C, IMG_H, IMG_W = 3, 32, 32
IMG_ELEMS = IMG_C * IMG_H * IMG_W

# Seeds of the five input streams (data, split, clustering, init, sampler).
SEED_DATA, SEED_SPLIT, SEED_CLUSTER, SEED_INIT, SEED_SAMPLER = 0, 1, 2, 3, 4


@dataclass
class Dataset:
    images: np.ndarray   # float32 [n, 3, 32, 32], NCHW
    labels: np.ndarray   # int32 [n]
    owner: np.ndarray    # int32 [n], client id of each example
    num_classes: int
    num_clients: int


def make_images(n: int, seed: int = SEED_DATA) -> np.ndarray:
    """n images of N(0,1) float32 pixels, NCHW."""
    rng = np.random.default_rng(seed)
    return rng.standard_normal((n, IMG_C, IMG_H, IMG_W), dtype=np.float32)


def make_labels(n: int, num_classes: int, balanced: bool, seed: int = SEED_DATA) -> np.ndarray:
    """Labels: exactly n/num_classes per class in shuffled order when
    `balanced`, otherwise i.i.d. uniform."""
    rng = np.random.default_rng(seed + 1_000_003)
    if balanced:
        if n % num_classes:
            raise ValueError("balanced labels need n divisible by num_classes")
        lab = np.repeat(np.arange(num_classes, dtype=np.int32), n // num_classes)
        rng.shuffle(lab)
        return lab
    return rng.integers(0, num_classes, size=n, dtype=np.int32)


def dirichlet_split(labels: np.ndarray, num_clients: int, alpha: float,
                    seed: int = SEED_SPLIT) -> np.ndarray:
    """Owner of every example under a per-class Dirichlet(alpha) split.

    For each class in increasing order: draw p ~ Dir(alpha * 1_K); give client
    k floor(p_k * n_class) examples; hand the remaining examples one each to the
    clients with the largest fractional parts (ties to the lower client id);
    shuffle the class's examples and deal them out in client order.  Clients
    may end up with no examples.
    """
    rng = np.random.default_rng(seed)
    owner = np.full(labels.shape[0], -1, dtype=np.int32)
    num_classes = int(labels.max()) + 1 if labels.size else 0
    for c in range(num_classes):
        ex = np.flatnonzero(labels == c)
        n_c = ex.size
        p = rng.dirichlet(np.full(num_clients, alpha))
        raw = p * n_c
        cnt = np.floor(raw).astype(np.int64)
        rem = n_c - int(cnt.sum())
        frac = raw - cnt
        # largest fractional part first, ties to the lower client id
        order = np.lexsort((np.arange(num_clients), -frac))
        cnt[order[:rem]] += 1
        rng.shuffle(ex)
        owner[ex] = np.repeat(np.arange(num_clients, dtype=np.int32), cnt)
    assert (owner >= 0).all()
    return owner


def class_support(num_clients: int, num_classes: int, per_client: int,
                  seed: int = SEED_SPLIT) -> np.ndarray:
    """[K][per_client] distinct classes of each client: client k's first is
    k mod num_classes (so every class has a holder once K >= num_classes),
    the others are drawn uniformly without replacement from the rest."""
    if not 1 <= per_client <= num_classes:
        raise ValueError("per_client must lie in [1, num_classes]")
    rng = np.random.default_rng(seed)
    sup = np.empty((num_clients, per_client), dtype=np.int32)
    for k in range(num_clients):
        first = k % num_classes
        rest = np.delete(np.arange(num_classes), first)
        sup[k, 0] = first
        sup[k, 1:] = rng.choice(rest, size=per_client - 1, replace=False)
    return sup


def extended_dirichlet_split(labels: np.ndarray, num_clients: int, per_client: int,
                             alpha: float, seed: int = SEED_SPLIT) -> np.ndarray:
    """Owner of every example under the extended-Dirichlet protocol of
    Section V-A: each client holds `per_client` classes (class_support), and
    each class's examples go to its holders in Dirichlet(alpha) proportions,
    dealt as in dirichlet_split (floor, largest remainders, shuffled deal).
    A class no client holds (K < num_classes) keeps owner -1 and is rejected."""
    num_classes = int(labels.max()) + 1 if labels.size else 0
    sup = class_support(num_clients, num_classes, per_client, seed)
    rng = np.random.default_rng(seed + 7_919)
    owner = np.full(labels.shape[0], -1, dtype=np.int32)
    for c in range(num_classes):
        holders = np.flatnonzero((sup == c).any(axis=1)).astype(np.int32)
        ex = np.flatnonzero(labels == c)
        if holders.size == 0:
            raise ValueError(f"class {c} has no holder")
        p = rng.dirichlet(np.full(holders.size, alpha))
        raw = p * ex.size
        cnt = np.floor(raw).astype(np.int64)
        rem = ex.size - int(cnt.sum())
        order = np.lexsort((np.arange(holders.size), -(raw - cnt)))
        cnt[order[:rem]] += 1
        rng.shuffle(ex)
        owner[ex] = np.repeat(holders, cnt)
    return owner


def make_dataset(n: int, num_classes: int, num_clients: int, alpha: float,
                 balanced: bool, seed_data: int = SEED_DATA,
                 seed_split: int = SEED_SPLIT, classes_per_client: int = 0) -> Dataset:
    """classes_per_client = 0: per-class Dirichlet(alpha) over all clients;
    m > 0: the extended-Dirichlet split with m classes per client."""
    images = make_images(n, seed_data)
    labels = make_labels(n, num_classes, balanced, seed_data)
    if classes_per_client:
        owner = extended_dirichlet_split(labels, num_clients, classes_per_client, alpha,
                                         seed_split)
    else:
        owner = dirichlet_split(labels, num_clients, alpha, seed_split)
    return Dataset(images, labels, owner, num_classes, num_clients)


# ---------------------------------------------------------------------------
# Split-model parameter shapes, in PyTorch state_dict order (conv weights
# OIHW), client segment first.  Conv layers are 3x3, stride 1, padding 1,
# with bias; every conv is followed by ReLU; `pool` adds a 2x2/2 max-pool.
# ---------------------------------------------------------------------------
ARCH_TINY_CNN, ARCH_SPLIT_CNN, ARCH_RESNET18, ARCH_RESNET18_C100 = 0, 1, 2, 3
RESNET_ARCHS = {ARCH_RESNET18: 10, ARCH_RESNET18_C100: 100}     # arch -> classes

ARCHS = {
    # (cin, cout, H, W, pool) per conv layer; fc (in, out)
    ARCH_TINY_CNN: dict(client=[(3, 16, 32, 32, 1)],
                        server=[(16, 32, 16, 16, 1)], fc=(2048, 10)),
    ARCH_SPLIT_CNN: dict(client=[(3, 32, 32, 32, 0), (32, 64, 32, 32, 1)],
                         server=[(64, 128, 16, 16, 1), (128, 128, 8, 8, 1)],
                         fc=(2048, 10)),
}


# The CIFAR ResNet-18 split: client = conv 3->64 stem + GroupNorm + stage 1,
# server = stages 2-4 with BatchNorm, global average pool, linear 512->J
# (J = 10, or 100 for ARCH_RESNET18_C100).
# Basic blocks (conv1, norm1, conv2, norm2[, shortcut conv 1x1, norm]);
# convolutions have no bias.  Names and order follow PyTorch's
# named_parameters() of the usual CIFAR ResNet-18 module layout.
RESNET_STAGES = ((64, 1), (128, 2), (256, 2), (512, 2))     # (width, first stride)


def _resnet_shapes(segment: str, classes: int):
    out = []
    if segment == "client":
        out += [("conv1.weight", (64, 3, 3, 3)), ("bn1.weight", (64,)), ("bn1.bias", (64,))]
    cin = 64
    for st, (width, stride) in enumerate(RESNET_STAGES):
        for j in range(2):
            s = stride if j == 0 else 1
            in_client = st == 0
            if (segment == "client") == in_client:
                pre = f"layer{st + 1}.{j}"
                out += [(f"{pre}.conv1.weight", (width, cin, 3, 3)),
                        (f"{pre}.bn1.weight", (width,)), (f"{pre}.bn1.bias", (width,)),
                        (f"{pre}.conv2.weight", (width, width, 3, 3)),
                        (f"{pre}.bn2.weight", (width,)), (f"{pre}.bn2.bias", (width,))]
                if s != 1 or cin != width:
                    out += [(f"{pre}.shortcut.0.weight", (width, cin, 1, 1)),
                            (f"{pre}.shortcut.1.weight", (width,)),
                            (f"{pre}.shortcut.1.bias", (width,))]
            cin = width
    if segment == "server":
        out += [("linear.weight", (classes, 512)), ("linear.bias", (classes,))]
    return out


def param_shapes(arch: int, segment: str):
    """[(name, shape)] for one segment ('client' or 'server')."""
    if arch in RESNET_ARCHS:
        return _resnet_shapes(segment, RESNET_ARCHS[arch])
    spec = ARCHS[arch]
    out = []
    for i, (cin, cout, _h, _w, _p) in enumerate(spec[segment]):
        out.append((f"{segment}.conv{i}.weight", (cout, cin, 3, 3)))
        out.append((f"{segment}.conv{i}.bias", (cout,)))
    if segment == "server":
        fin, fout = spec["fc"]
        out.append(("server.fc.weight", (fout, fin)))
        out.append(("server.fc.bias", (fout,)))
    return out


def num_classes(arch: int) -> int:
    return RESNET_ARCHS.get(arch, 10)


def num_params(arch: int, segment: str) -> int:
    return int(sum(np.prod(s) for _n, s in param_shapes(arch, segment)))


def init_params(arch: int, seed: int = SEED_INIT) -> np.ndarray:
    """One float32 blob, client segment then server segment, drawn like
    PyTorch's default layer init: U(-1/sqrt(fan_in), 1/sqrt(fan_in)) for
    weights and biases of every conv and linear layer."""
    rng = np.random.default_rng(seed)
    parts = []
    for seg in ("client", "server"):
        shapes = param_shapes(arch, seg)
        for (name, shape) in shapes:
            if len(shape) == 1 and (".bn" in name or "shortcut.1" in name or
                                    name.startswith("bn1")):
                # norm affine: weight 1, bias 0 (PyTorch's default)
                val = 1.0 if name.endswith(".weight") else 0.0
                parts.append(np.full(shape, val, dtype=np.float32))
                continue
            if name.endswith(".weight"):
                fan_in = int(np.prod(shape[1:]))
            bound = 1.0 / np.sqrt(fan_in)
            parts.append(rng.uniform(-bound, bound, size=shape).astype(np.float32).ravel())
    return np.concatenate(parts)
