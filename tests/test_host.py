"""Host-side checks that need no GPU: the library loads and exports every
entry point of include/gcpsl.h, gcpsl_init rejects bad arguments before it
touches the device, the product never imports the oracle, and the clustering
rules of Algorithm 1 behave as stated."""
import ctypes as ct
import os
import re

import numpy as np
import pytest

import paper_2609_29395_gb300 as pkg
from paper_2609_29395_gb300 import binding, clustering, configs, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_29395_gb300 import build
    build.build()
    return binding.load()


def test_header_declares_what_the_library_exports(lib):
    hdr = open(os.path.join(ROOT, "include", "gcpsl.h")).read()
    declared = set(re.findall(r"\b(gcpsl_[a-z_]+)\s*\(", hdr))
    assert declared == set(binding.EXPORTS)
    for name in declared:
        assert hasattr(lib, name), name


def test_num_params(lib):
    assert pkg.gcpsl_num_params(binding.GCPSL_SPLIT_CNN, 0) + \
        pkg.gcpsl_num_params(binding.GCPSL_SPLIT_CNN, 1) == 261_322
    assert pkg.gcpsl_num_params(binding.GCPSL_TINY_CNN, 0) + \
        pkg.gcpsl_num_params(binding.GCPSL_TINY_CNN, 1) == 25_578
    assert pkg.gcpsl_num_params(binding.GCPSL_SPLIT_CNN, 0) == synth.num_params(1, "client")
    assert pkg.gcpsl_num_params(7, 0) == -1
    # the 100-way head adds 90 rows of 512 weights and 90 biases to the server
    for seg in (0, 1):
        assert pkg.gcpsl_num_params(binding.GCPSL_RESNET18_C100, seg) == \
            synth.num_params(synth.ARCH_RESNET18_C100, ("client", "server")[seg])
    assert pkg.gcpsl_num_params(binding.GCPSL_RESNET18_C100, 1) - \
        pkg.gcpsl_num_params(binding.GCPSL_RESNET18, 1) == 90 * 513
    assert pkg.gcpsl_num_params(binding.GCPSL_RESNET18_C100, 0) == \
        pkg.gcpsl_num_params(binding.GCPSL_RESNET18, 0)


def _ds(n=256, K=8):
    return synth.make_dataset(n, 10, K, 0.5, balanced=False)


def test_binding_structs_follow_the_header():
    """The ctypes mirrors list the header's struct members in order."""
    hdr = open(os.path.join(ROOT, "include", "gcpsl.h")).read()
    for struct, cls in (("gcpsl_model_desc", binding.gcpsl_model_desc),
                        ("gcpsl_dataset", binding.gcpsl_dataset)):
        body = re.search(r"typedef struct \{([^{}]*)\}\s*" + struct + ";", hdr).group(1)
        body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
        names = []
        for decl in body.split(";"):
            decl = decl.strip()
            if not decl:
                continue
            # "float lr, momentum, weight_decay" / "const float* images"
            parts = [p.strip() for p in decl.split(",")]
            names.append(re.findall(r"(\w+)\s*$", parts[0])[0])
            names += [p.strip("* ") for p in parts[1:]]
        assert names == [f[0] for f in cls._fields_], (struct, names)


@pytest.mark.parametrize("case", ["small_cluster", "assign_range", "owner_range", "label_range",
                                  "bad_B", "bad_arch", "bad_dtype", "class_count", "gn_groups",
                                  "bn_momentum"])
def test_init_rejects_bad_arguments(lib, case):
    ds = _ds()
    K, C, B = 8, 2, 16
    assign = clustering.random_clustering(K, C, 0)
    kw = dict(arch=0, K=K, C=C, assignment=assign, B=B, F=0, seed=1, images=ds.images,
              labels=ds.labels, owner=ds.owner)
    if case == "small_cluster":
        kw["B"] = 1000
    elif case == "assign_range":
        kw["assignment"] = np.full(K, 2, np.int32)
    elif case == "owner_range":
        kw["owner"] = np.where(np.arange(ds.owner.size) == 3, K, ds.owner).astype(np.int32)
    elif case == "label_range":
        kw["labels"] = np.where(np.arange(ds.labels.size) == 5, 10, ds.labels).astype(np.int32)
    elif case == "bad_B":
        kw["B"] = 0
    elif case == "bad_arch":
        kw["arch"] = 9
    elif case == "gn_groups":
        kw["gn_groups"] = 3             # does not divide the 64 GroupNorm channels
    elif case == "bn_momentum":
        kw["bn_momentum"] = 1.5
    with pytest.raises(binding.GcpslError) as e:
        if case == "class_count":
            # a 10-class dataset declared to a 100-class architecture
            desc = binding.gcpsl_model_desc(binding.GCPSL_RESNET18_C100, 1, 0.05, 0, 0, 0, 0, 0,
                                            0, 0)
            ds_c = binding.gcpsl_dataset(binding._p(ds.images, ct.c_float),
                                         binding._p(ds.labels, ct.c_int32),
                                         binding._p(ds.owner, ct.c_int32), ds.images.shape[0], 10)
            h = ct.c_void_p()
            st = lib.gcpsl_init(ct.byref(desc), K, C, binding._p(assign, ct.c_int32), B, 0, 1,
                                ct.byref(ds_c), None, ct.byref(h))
            binding._check(st)
        elif case == "bad_dtype":
            desc = binding.gcpsl_model_desc(0, 7, 0.05, 0, 0, 0, 0, 0, 0, 0)
            ds_c = binding.gcpsl_dataset(binding._p(ds.images, ct.c_float),
                                         binding._p(ds.labels, ct.c_int32),
                                         binding._p(ds.owner, ct.c_int32), ds.images.shape[0], 10)
            h = ct.c_void_p()
            st = lib.gcpsl_init(ct.byref(desc), K, C, binding._p(assign, ct.c_int32), B, 0, 1,
                                ct.byref(ds_c), None, ct.byref(h))
            binding._check(st)
        else:
            binding.Context(**kw)
    want = binding.GCPSL_E_UNSUPPORTED if case == "bad_arch" else binding.GCPSL_E_INVAL
    assert e.value.status == want
    assert lib.gcpsl_last_error(None)


def test_product_never_touches_the_oracle():
    pat = re.compile(r"^\s*(import|from)\s+oracle\b|oracle/|gcpsl_oracle", re.M)
    for dirpath, _dirs, files in os.walk(os.path.join(ROOT, "paper_2609_29395_gb300")):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                src = open(os.path.join(dirpath, f)).read()
                assert not pat.search(src), f


# --------------------------------------------------------------------------
# Algorithm 1 rules
# --------------------------------------------------------------------------
def test_random_clustering_round_robin():
    a = clustering.random_clustering(37, 5, 3)
    card = np.bincount(a, minlength=5)
    assert card.max() - card.min() <= 1 and card.sum() == 37
    assert (a == clustering.random_clustering(37, 5, 3)).all()


def test_size_balanced_greedy_rule():
    rng = np.random.default_rng(0)
    sizes = rng.integers(0, 500, size=23)
    C = 4
    a = clustering.size_balanced_clustering(sizes, C)
    cap = -(-23 // C)
    assert np.bincount(a, minlength=C).max() <= cap
    # replay: every client went to the lightest allowed cluster at its turn
    order = sorted(range(23), key=lambda k: (-sizes[k], k))
    load, card = np.zeros(C), np.zeros(C, int)
    for k in order:
        allowed = [n for n in range(C) if card[n] < cap]
        assert a[k] == min(allowed, key=lambda n: (load[n], n))
        load[a[k]] += sizes[k]
        card[a[k]] += 1
    rnd = clustering.random_clustering(23, C, 0)
    spread = lambda asg: np.ptp(np.bincount(asg, weights=sizes, minlength=C))
    assert spread(a) <= spread(rnd)


def test_label_aware_greedy_is_closer_to_global():
    ds = synth.make_dataset(4000, 10, 64, 0.3, balanced=True)
    hist = clustering.client_histograms(ds.owner, ds.labels, 64, 10)
    glob = hist.sum(0) / hist.sum()

    def mean_l1(asg):
        d = []
        for n in range(8):
            h = hist[asg == n].sum(0)
            d.append(np.abs(h / h.sum() - glob).sum())
        return np.mean(d)
    la = clustering.label_aware_greedy(hist, 8)
    assert np.bincount(la, minlength=8).max() <= 8
    assert mean_l1(la) < mean_l1(clustering.random_clustering(64, 8, 0))


def test_objective_j_by_hand():
    # two clusters, two classes: cluster 0 = [3, 1], cluster 1 = [1, 3]
    hist = np.array([[3, 1], [1, 3]])
    j = clustering.objective_j(hist, np.array([0, 1]), 2)
    p, pn = np.array([0.5, 0.5]), np.array([0.75, 0.25])
    m = 0.5 * (p + pn)
    jsd = 0.5 * np.sum(pn * np.log(pn / m)) + 0.5 * np.sum(p * np.log(p / m))
    assert j == pytest.approx(0.0 + 2 * 0.5 * jsd, rel=1e-12)
    assert clustering.objective_j(hist, np.array([0, 0]), 2) == pytest.approx(1.0)


def test_label_aware_local_search_reaches_local_optimum():
    rng = np.random.default_rng(1)
    hist = rng.integers(0, 20, size=(10, 3))
    C = 3
    a = clustering.label_aware_local_search(hist, C)
    j = clustering.objective_j(hist, a, C)
    assert j <= clustering.objective_j(hist, clustering.size_balanced_clustering(hist.sum(1), C), C)
    cap = -(-10 // C)
    card = np.bincount(a, minlength=C)
    for k in range(10):
        for n in range(C):
            if n == a[k] or card[n] >= cap:
                continue
            b = a.copy()
            b[k] = n
            assert clustering.objective_j(hist, b, C) >= j - 1e-12


def test_workloads_fit_their_batch():
    w = configs.WORKLOADS["tiny"]
    ds, assign, params = configs.build_inputs(w)
    sizes = configs.cluster_sizes(ds.owner, assign, w.num_clusters)
    assert (sizes >= w.B).all()
    assert params.size == synth.num_params(w.arch, "client") + synth.num_params(w.arch, "server")


# --------------------------------------------------------------------------
# Extended-Dirichlet client split (Section V-A)
# --------------------------------------------------------------------------
def test_class_support_covers_every_class():
    sup = synth.class_support(256, 100, 2, seed=5)
    assert sup.shape == (256, 2)
    assert (sup[:, 0] == np.arange(256) % 100).all()
    assert (sup[:, 0] != sup[:, 1]).all()
    assert set(np.unique(sup)) == set(range(100))
    # the second class is uniform over the other 99: chi-square over 256 draws
    # is loose, so check only the range and that many classes appear
    assert len(np.unique(sup[:, 1])) > 80
    with pytest.raises(ValueError):
        synth.class_support(8, 10, 0)


def test_extended_dirichlet_split_invariants():
    n, J, K, m = 20_000, 100, 256, 2
    labels = synth.make_labels(n, J, True)
    owner = synth.extended_dirichlet_split(labels, K, m, 3.0, seed=9)
    sup = synth.class_support(K, J, m, seed=9)
    assert owner.shape == labels.shape and owner.min() >= 0 and owner.max() < K
    # every example's class is one of its owner's classes
    assert (sup[owner] == labels[:, None]).any(axis=1).all()
    # every class's examples all went to its holders, and were all dealt
    for c in (0, 17, 99):
        holders = set(np.flatnonzero((sup == c).any(axis=1)))
        assert set(np.unique(owner[labels == c])) <= holders
    assert np.bincount(labels, minlength=J).sum() == n
    # deterministic
    assert (owner == synth.extended_dirichlet_split(labels, K, m, 3.0, seed=9)).all()


def test_extended_dirichlet_concentration():
    """Large alpha spreads a class evenly over its holders; small alpha
    concentrates it (Dirichlet concentration)."""
    labels = synth.make_labels(100_000, 10, True)
    spread = {}
    for alpha in (1000.0, 0.05):
        owner = synth.extended_dirichlet_split(labels, 40, 2, alpha, seed=3)
        sup = synth.class_support(40, 10, 2, seed=3)
        cv = []
        for c in range(10):
            holders = np.flatnonzero((sup == c).any(axis=1))
            cnt = np.bincount(owner[labels == c], minlength=40)[holders]
            cv.append(cnt.std() / cnt.mean())
        spread[alpha] = float(np.mean(cv))
    assert spread[1000.0] < 0.1 < 1.0 < spread[0.05]


def test_cifar100_workload_inputs():
    w = configs.WORKLOADS["resnet18_c100_c4"]
    assert w.num_classes == 100
    ds, assign, params = configs.build_inputs(w)
    assert ds.num_classes == 100 and ds.labels.max() == 99
    assert np.bincount(ds.labels).min() == np.bincount(ds.labels).max() == 500
    per_client = [np.unique(ds.labels[ds.owner == k]).size for k in range(w.num_clients)]
    assert max(per_client) <= 2
    sizes = configs.cluster_sizes(ds.owner, assign, w.num_clusters)
    assert (sizes >= w.B).all() and sizes.sum() == w.n
    assert params.size == synth.num_params(w.arch, "client") + synth.num_params(w.arch, "server")
