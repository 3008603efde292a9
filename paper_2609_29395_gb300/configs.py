"""The five synthetic GCPSL workloads (images 32x32x3, N(0,1) pixels, 10
classes) and the host-side recipe that builds their inputs.

Each workload fixes the dataset size, the client split, the clustering rule,
the per-workload batch B, the fusion interval F (in steps), the split model
and the optimiser.  `build_inputs` returns everything `gcpsl_init` takes.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

from . import clustering, synth


@dataclass
class Workload:
    name: str
    n: int
    num_clients: int
    alpha: float
    balanced_labels: bool
    num_clusters: int
    rule: str          # 'random' | 'size' | 'label_greedy' | 'label_search'
    B: int
    F: int
    arch: int
    bf16: bool
    lr: float = 0.05
    momentum: float = 0.0
    steps: int = 10
    extra: dict = field(default_factory=dict)


WORKLOADS = {
    "tiny": Workload("tiny", 512, 16, 0.5, False, 2, "random", 32, 5,
                     synth.ARCH_TINY_CNN, False, 0.05, 0.0, 10),
    "splitcnn_c4": Workload("splitcnn_c4", 50_000, 256, 0.3, True, 4, "random", 64, 50,
                            synth.ARCH_SPLIT_CNN, True, 0.05, 0.9),
    "splitcnn_c16": Workload("splitcnn_c16", 50_000, 256, 0.3, True, 16, "size", 64, 50,
                             synth.ARCH_SPLIT_CNN, True, 0.05, 0.9),
    "splitcnn_c64": Workload("splitcnn_c64", 50_000, 256, 0.3, True, 64, "label_greedy", 64, 25,
                             synth.ARCH_SPLIT_CNN, True, 0.05, 0.9),
    # 200,000 images (20,000 per class), K = 1024, Dir(0.1), C = 8 random,
    # B = 128, F = 100, the ResNet-18 split
    "resnet18_c8": Workload("resnet18_c8", 200_000, 1024, 0.1, True, 8, "random", 128, 100,
                            synth.ARCH_RESNET18, True, 0.05, 0.9),
}


def assign_clusters(w: Workload, ds: synth.Dataset) -> np.ndarray:
    k = w.num_clients
    if w.rule == "random":
        return clustering.random_clustering(k, w.num_clusters, synth.SEED_CLUSTER)
    if w.rule == "size":
        return clustering.size_balanced_clustering(
            clustering.client_counts(ds.owner, k), w.num_clusters)
    hist = clustering.client_histograms(ds.owner, ds.labels, k, ds.num_classes)
    if w.rule == "label_greedy":
        return clustering.label_aware_greedy(hist, w.num_clusters)
    if w.rule == "label_search":
        return clustering.label_aware_local_search(hist, w.num_clusters)
    raise ValueError(w.rule)


def build_inputs(w: Workload):
    """(dataset, assignment int32[K], init_params float32[P]) for a workload."""
    ds = synth.make_dataset(w.n, 10, w.num_clients, w.alpha, w.balanced_labels)
    assign = assign_clusters(w, ds)
    params = synth.init_params(w.arch)
    return ds, assign, params


def cluster_sizes(owner: np.ndarray, assign: np.ndarray, num_clusters: int) -> np.ndarray:
    return np.bincount(assign[owner], minlength=num_clusters)
