"""Static client clustering (Algorithm 1, Section IV-A).

Host-side setup that runs once before training; its output, the fixed
client -> cluster map, is an input of `gcpsl_init`.  Three rules:

* random: permute the clients, deal them round-robin (no metadata).
* size-balanced: sort clients by decreasing sample count, place each in the
  allowed cluster with the smallest current sample count.
* label-aware: uses per-client class histograms.  `label_aware_greedy` is the
  one-pass greedy rule (minimise the l1 distance of the cluster's label
  distribution to the global one); `label_aware_local_search` is the paper's
  single-client-move search on J (Eq. 4).

"Allowed" means the cluster holds fewer than ceil(K/N) clients (the paper's
maximum cluster cardinality, whose value it does not state).  All ties go to
the lowest cluster index, so every rule is deterministic.
"""
from __future__ import annotations

import numpy as np


def client_counts(owner: np.ndarray, num_clients: int) -> np.ndarray:
    return np.bincount(owner, minlength=num_clients).astype(np.int64)


def client_histograms(owner: np.ndarray, labels: np.ndarray, num_clients: int,
                      num_classes: int) -> np.ndarray:
    h = np.zeros((num_clients, num_classes), dtype=np.int64)
    np.add.at(h, (owner, labels), 1)
    return h


def random_clustering(num_clients: int, num_clusters: int, seed: int) -> np.ndarray:
    """Algorithm 1, random rule: permute, then assign round-robin."""
    perm = np.random.default_rng(seed).permutation(num_clients)
    assign = np.empty(num_clients, dtype=np.int32)
    assign[perm] = np.arange(num_clients) % num_clusters
    return assign


def _size_order(sizes: np.ndarray) -> np.ndarray:
    # decreasing sample count, ties to the lower client id
    return np.lexsort((np.arange(sizes.size), -sizes))


def size_balanced_clustering(sizes: np.ndarray, num_clusters: int) -> np.ndarray:
    """Algorithm 1, size-balanced rule."""
    k = sizes.size
    cap = -(-k // num_clusters)
    load = np.zeros(num_clusters, dtype=np.int64)
    card = np.zeros(num_clusters, dtype=np.int64)
    assign = np.empty(k, dtype=np.int32)
    for cl in _size_order(sizes):
        allowed = np.flatnonzero(card < cap)
        n = allowed[np.argmin(load[allowed])]   # argmin keeps the lowest index
        assign[cl] = n
        load[n] += sizes[cl]
        card[n] += 1
    return assign


def label_aware_greedy(hist: np.ndarray, num_clusters: int) -> np.ndarray:
    """One-pass label-aware rule: in decreasing-size order, put each client in
    the allowed cluster whose label distribution after adding it is closest in
    l1 to the global distribution.  An empty histogram normalises to zero."""
    k, _ = hist.shape
    sizes = hist.sum(1)
    glob = hist.sum(0) / max(1, hist.sum())
    cap = -(-k // num_clusters)
    acc = np.zeros((num_clusters, hist.shape[1]), dtype=np.int64)
    card = np.zeros(num_clusters, dtype=np.int64)
    assign = np.empty(k, dtype=np.int32)
    for cl in _size_order(sizes):
        best, best_d = -1, np.inf
        for n in range(num_clusters):
            if card[n] >= cap:
                continue
            h = acc[n] + hist[cl]
            tot = h.sum()
            d = np.abs((h / tot if tot else h.astype(np.float64)) - glob).sum()
            if d < best_d:
                best, best_d = n, d
        assign[cl] = best
        acc[best] += hist[cl]
        card[best] += 1
    return assign


def _jsd(p: np.ndarray, q: np.ndarray) -> float:
    m = 0.5 * (p + q)
    def kl(a, b):
        nz = a > 0
        return float(np.sum(a[nz] * np.log(a[nz] / b[nz])))
    return 0.5 * kl(p, m) + 0.5 * kl(q, m)


def objective_j(hist: np.ndarray, assign: np.ndarray, num_clusters: int) -> float:
    """Eq. 4: sum_n |w_n - wbar| / |D| + sum_n (w_n/|D|) JSD(p_n, p)."""
    total = hist.sum()
    glob = hist.sum(0) / total
    wbar = total / num_clusters
    j = 0.0
    for n in range(num_clusters):
        h = hist[assign == n].sum(0)
        w = h.sum()
        j += abs(w - wbar) / total
        if w:
            j += (w / total) * _jsd(h / w, glob)
    return j


def label_aware_local_search(hist: np.ndarray, num_clusters: int,
                             max_moves: int = 10_000) -> np.ndarray:
    """Algorithm 1, label-aware branch: start from the size-balanced
    assignment and apply the best improving single-client move (allowed =
    target below the cardinality cap) until none improves J or the move
    limit is reached."""
    k = hist.shape[0]
    cap = -(-k // num_clusters)
    assign = size_balanced_clustering(hist.sum(1), num_clusters)
    cur = objective_j(hist, assign, num_clusters)
    for _ in range(max_moves):
        card = np.bincount(assign, minlength=num_clusters)
        best = (cur, -1, -1)
        for cl in range(k):
            src = assign[cl]
            for n in range(num_clusters):
                if n == src or card[n] >= cap:
                    continue
                assign[cl] = n
                v = objective_j(hist, assign, num_clusters)
                assign[cl] = src
                if v < best[0] - 1e-15:
                    best = (v, cl, n)
        if best[1] < 0:
            break
        cur, cl, n = best
        assign[cl] = n
    return assign


def schedule_rounds(sizes: np.ndarray, B: int) -> np.ndarray:
    """r_n = n_c // B local rounds per epoch of each cluster (Section IV-C)."""
    return np.asarray(sizes, dtype=np.int64) // B


def ideal_schedule_speedup(sizes: np.ndarray, B: int):
    """Eq. 6: S_ideal = sum_n r_n / max_n r_n and E_ideal = S_ideal / N for
    one epoch of the concurrent schedule (clusters with fewer rounds wait at
    the fusion barrier)."""
    r = schedule_rounds(sizes, B)
    s = float(r.sum()) / float(r.max())
    return s, s / r.size

