"""The synthetic GCPSL workloads (images 32x32x3, N(0,1) pixels, 10 or 100
classes) and the host-side recipe that builds their inputs.

Each workload fixes the dataset size, the client split, the clustering rule,
the per-workload batch B, the fusion interval F (in steps), the split model
and the optimiser.  `build_inputs` returns everything `gcpsl_init` takes and
`Workload.options()` the optimiser / augmentation keywords of `Context`.
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
    weight_decay: float = 0.0
    nesterov: bool = False
    label_smoothing: float = 0.0
    augment: bool = False
    classes_per_client: int = 0   # > 0: the extended-Dirichlet split of Section V-A

    @property
    def num_classes(self) -> int:
        return synth.num_classes(self.arch)

    def options(self) -> dict:
        """Optimiser and augmentation keywords of Context / Oracle."""
        return dict(lr=self.lr, momentum=self.momentum, weight_decay=self.weight_decay,
                    nesterov=self.nesterov, label_smoothing=self.label_smoothing,
                    augment=self.augment)


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
    # The CIFAR-100 shape of Section V-A: 50,000 images (500 per class, 100
    # classes), K = 256 clients holding two classes each (extended Dirichlet,
    # alpha = 3), C = 4 label-aware clusters (the JSD local search of Eq. 4),
    # B = 128, 100-step fusion, the ResNet-18 split with a 100-way head and the
    # paper's training recipe (lr 0.01, Nesterov momentum 0.9, weight decay
    # 5e-4, label smoothing 0.1, random crop + flip)
    "resnet18_c100_c4": Workload("resnet18_c100_c4", 50_000, 256, 3.0, True, 4, "label_search",
                                 128, 100, synth.ARCH_RESNET18_C100, True, 0.01, 0.9,
                                 weight_decay=5e-4, nesterov=True, label_smoothing=0.1,
                                 augment=True, classes_per_client=2),
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
    ds = synth.make_dataset(w.n, w.num_classes, w.num_clients, w.alpha, w.balanced_labels,
                            classes_per_client=w.classes_per_client)
    assign = assign_clusters(w, ds)
    params = synth.init_params(w.arch)
    return ds, assign, params


def cluster_sizes(owner: np.ndarray, assign: np.ndarray, num_clusters: int) -> np.ndarray:
    return np.bincount(assign[owner], minlength=num_clusters)
