"""Thin ctypes binding of libgcpsl.so: the C ABI of include/gcpsl.h under the
same names, plus a small `Context` class that marshals numpy arrays.

Nothing here computes any part of the training step; every step runs in the
library's CUDA kernels.  Loading fails loudly when the library has not been
built (there is no fallback).
"""
from __future__ import annotations

import ctypes as ct
from pathlib import Path

import numpy as np

LIB_PATH = Path(__file__).resolve().parent / "lib" / "libgcpsl.so"

GCPSL_OK, GCPSL_E_INVAL, GCPSL_E_NOMEM, GCPSL_E_CUDA, GCPSL_E_STATE, GCPSL_E_TIMEOUT, \
    GCPSL_E_UNSUPPORTED = range(7)
GCPSL_TINY_CNN, GCPSL_SPLIT_CNN, GCPSL_RESNET18, GCPSL_RESNET18_C100 = 0, 1, 2, 3
GCPSL_F32, GCPSL_BF16 = 0, 1
GCPSL_CLIENT, GCPSL_SERVER, GCPSL_BN_STATE = 0, 1, 2
GCPSL_CUT_ACT, GCPSL_CUT_GRAD = 0, 1

STATUS_NAMES = {0: "OK", 1: "E_INVAL", 2: "E_NOMEM", 3: "E_CUDA", 4: "E_STATE", 5: "E_TIMEOUT",
                6: "E_UNSUPPORTED"}

# every entry point declared in include/gcpsl.h
EXPORTS = ("gcpsl_init", "gcpsl_step", "gcpsl_fuse", "gcpsl_get_params", "gcpsl_set_params",
           "gcpsl_set_bn_state", "gcpsl_get_relu_masks",
           "gcpsl_get_momentum", "gcpsl_set_momentum", "gcpsl_get_pool_codes",
           "gcpsl_get_cut", "gcpsl_cut_elems", "gcpsl_get_sample", "gcpsl_num_params",
           "gcpsl_rounds", "gcpsl_set_stream", "gcpsl_set_graph", "gcpsl_set_timing",
           "gcpsl_set_timing_filter", "gcpsl_kernels_launched",
           "gcpsl_kernel_times",
           "gcpsl_reset_kernel_times", "gcpsl_sample_round_noalloc",
           "gcpsl_check_wait_timeout", "gcpsl_last_error", "gcpsl_destroy")


class gcpsl_model_desc(ct.Structure):
    _fields_ = [("arch", ct.c_int), ("operand_dtype", ct.c_int), ("lr", ct.c_float),
                ("momentum", ct.c_float), ("weight_decay", ct.c_float), ("nesterov", ct.c_int),
                ("label_smoothing", ct.c_float), ("cluster_id_base", ct.c_int),
                ("data_on_host", ct.c_int), ("augment", ct.c_int), ("gn_groups", ct.c_int),
                ("bn_momentum", ct.c_float), ("norm_eps", ct.c_float),
                ("client_average", ct.c_int)]


class gcpsl_dataset(ct.Structure):
    _fields_ = [("images", ct.POINTER(ct.c_float)), ("labels", ct.POINTER(ct.c_int32)),
                ("owner", ct.POINTER(ct.c_int32)), ("n", ct.c_int64), ("num_classes", ct.c_int)]


class gcpsl_step_stats(ct.Structure):
    _fields_ = [("loss", ct.POINTER(ct.c_float)), ("active", ct.POINTER(ct.c_int32))]


class GcpslError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


_lib = None


def load() -> ct.CDLL:
    """Load libgcpsl.so (built by paper_2609_29395_gb300.build)."""
    global _lib
    if _lib is not None:
        return _lib
    if not LIB_PATH.exists():
        raise ImportError(f"{LIB_PATH} is missing: build it with paper_2609_29395_gb300.build.build()")
    L = ct.CDLL(str(LIB_PATH))
    vp, i32p, f32p = ct.c_void_p, ct.POINTER(ct.c_int32), ct.POINTER(ct.c_float)
    L.gcpsl_init.argtypes = [ct.POINTER(gcpsl_model_desc), ct.c_int, ct.c_int, i32p, ct.c_int,
                             ct.c_int, ct.c_uint64, ct.POINTER(gcpsl_dataset), f32p,
                             ct.POINTER(vp)]
    L.gcpsl_step.argtypes = [vp, ct.POINTER(gcpsl_step_stats)]
    L.gcpsl_fuse.argtypes = [vp]
    L.gcpsl_get_params.argtypes = [vp, ct.c_int, ct.c_int, f32p, ct.c_size_t,
                                   ct.POINTER(ct.c_size_t)]
    L.gcpsl_set_params.argtypes = [vp, ct.c_int, f32p, ct.c_size_t]
    L.gcpsl_get_momentum.argtypes = [vp, ct.c_int, f32p, ct.c_size_t]
    L.gcpsl_set_momentum.argtypes = [vp, ct.c_int, f32p, ct.c_size_t]
    L.gcpsl_get_pool_codes.argtypes = [vp, ct.c_int, ct.POINTER(ct.c_uint8), ct.c_size_t]
    L.gcpsl_get_cut.argtypes = [vp, ct.c_int, f32p, ct.c_size_t]
    L.gcpsl_cut_elems.argtypes = [vp]
    L.gcpsl_cut_elems.restype = ct.c_size_t
    L.gcpsl_get_sample.argtypes = [vp, i32p, i32p]
    L.gcpsl_num_params.argtypes = [ct.c_int, ct.c_int]
    L.gcpsl_num_params.restype = ct.c_int64
    L.gcpsl_rounds.argtypes = [vp]
    L.gcpsl_rounds.restype = ct.c_int64
    L.gcpsl_set_stream.argtypes = [vp, vp]
    L.gcpsl_set_timing.argtypes = [vp, ct.c_int]
    L.gcpsl_set_graph.argtypes = [vp, ct.c_int]
    L.gcpsl_check_wait_timeout.argtypes = [vp, ct.c_uint64]
    L.gcpsl_set_bn_state.argtypes = [vp, ct.c_int, f32p, ct.c_size_t]
    L.gcpsl_get_relu_masks.argtypes = [vp, ct.POINTER(ct.c_uint8), ct.c_size_t,
                                       ct.POINTER(ct.c_size_t)]
    L.gcpsl_set_timing_filter.argtypes = [vp, ct.c_char_p]
    L.gcpsl_kernels_launched.argtypes = [vp]
    L.gcpsl_kernels_launched.restype = ct.c_int64
    L.gcpsl_kernel_times.argtypes = [vp, ct.POINTER(ct.c_char_p), ct.POINTER(ct.c_int64),
                                     ct.POINTER(ct.c_double), ct.c_int]
    L.gcpsl_kernel_times.restype = ct.c_int
    L.gcpsl_reset_kernel_times.argtypes = [vp]
    L.gcpsl_reset_kernel_times.restype = None
    L.gcpsl_sample_round_noalloc.argtypes = [vp, ct.POINTER(ct.c_int64), vp, vp, ct.c_int,
                                             ct.c_int, ct.c_int, ct.c_int64, ct.c_int,
                                             ct.c_uint64, vp, vp, vp, vp, vp]
    L.gcpsl_sample_round_noalloc.restype = ct.c_int
    L.gcpsl_last_error.argtypes = [vp]
    L.gcpsl_last_error.restype = ct.c_char_p
    L.gcpsl_destroy.argtypes = [vp]
    L.gcpsl_destroy.restype = None
    for name in ("gcpsl_init", "gcpsl_step", "gcpsl_fuse", "gcpsl_get_params", "gcpsl_set_params",
                 "gcpsl_get_cut", "gcpsl_get_sample", "gcpsl_set_stream", "gcpsl_set_timing",
                 "gcpsl_set_graph", "gcpsl_set_timing_filter", "gcpsl_set_bn_state",
                 "gcpsl_get_relu_masks",
                 "gcpsl_get_momentum", "gcpsl_set_momentum", "gcpsl_get_pool_codes"):
        getattr(L, name).restype = ct.c_int
    _lib = L
    return L


def _p(a, t):
    return a.ctypes.data_as(ct.POINTER(t))


def _check(st, h=None):
    if st != GCPSL_OK:
        msg = load().gcpsl_last_error(h)
        raise GcpslError(st, msg.decode() if msg else "")


# C-ABI names, argument marshalling only ----------------------------------
def num_classes(arch: int) -> int:
    """Classes of an architecture's linear head (the dataset's num_classes)."""
    return 100 if arch == GCPSL_RESNET18_C100 else 10


def gcpsl_num_params(arch: int, segment: int) -> int:
    return int(load().gcpsl_num_params(arch, segment))


def gcpsl_sample_round_noalloc(ids_dev: int, cluster_offsets, owner_dev: int, labels_dev: int,
                               K: int, C: int, B: int, round_: int, cluster_id_base: int,
                               seed: int, idx_dev: int, counts_dev: int, active_dev: int,
                               batch_labels_dev: int, stream: int | None = None):
    """The round sampler without device allocation; *_dev are device
    addresses (e.g. tensor.data_ptr()), cluster_offsets a host int64 array."""
    off = np.ascontiguousarray(cluster_offsets, dtype=np.int64)
    st = load().gcpsl_sample_round_noalloc(
        ct.c_void_p(ids_dev), _p(off, ct.c_int64), ct.c_void_p(owner_dev),
        ct.c_void_p(labels_dev), K, C, B, round_, cluster_id_base, seed, ct.c_void_p(idx_dev),
        ct.c_void_p(counts_dev), ct.c_void_p(active_dev), ct.c_void_p(batch_labels_dev),
        ct.c_void_p(stream) if stream else None)
    _check(st, None)


class Context:
    """One GCPSL context: C cluster workloads on the current GPU."""

    def __init__(self, arch, K, C, assignment, B, F, seed, images, labels, owner,
                 init_params=None, lr=0.05, momentum=0.0, weight_decay=0.0, nesterov=False,
                 label_smoothing=0.0, bf16=True, cluster_id_base=0, data_on_host=False,
                 augment=False, gn_groups=32, norm_eps=1e-5, bn_momentum=0.1,
                 client_average=False):
        L = load()
        self.K, self.C, self.B, self.arch = K, C, B, arch
        desc = gcpsl_model_desc(arch, GCPSL_BF16 if bf16 else GCPSL_F32, lr, momentum,
                                weight_decay, int(nesterov), label_smoothing, cluster_id_base,
                                int(data_on_host), int(augment), gn_groups, bn_momentum,
                                norm_eps, int(client_average))
        images = np.ascontiguousarray(images, dtype=np.float32)
        labels = np.ascontiguousarray(labels, dtype=np.int32)
        owner = np.ascontiguousarray(owner, dtype=np.int32)
        assignment = np.ascontiguousarray(assignment, dtype=np.int32)
        ds = gcpsl_dataset(_p(images, ct.c_float), _p(labels, ct.c_int32),
                           _p(owner, ct.c_int32), images.shape[0], num_classes(arch))
        init = None
        if init_params is not None:
            init = np.ascontiguousarray(init_params, dtype=np.float32)
        h = ct.c_void_p()
        st = L.gcpsl_init(ct.byref(desc), K, C, _p(assignment, ct.c_int32), B, F, seed,
                          ct.byref(ds), _p(init, ct.c_float) if init is not None else None,
                          ct.byref(h))
        _check(st, None)
        self._h = h
        self.P_client = gcpsl_num_params(arch, GCPSL_CLIENT)
        self.P_server = gcpsl_num_params(arch, GCPSL_SERVER)
        self._loss = np.zeros(C, dtype=np.float32)
        self._active = np.zeros(C, dtype=np.int32)
        self._stats = gcpsl_step_stats(_p(self._loss, ct.c_float), _p(self._active, ct.c_int32))

    def close(self):
        if getattr(self, "_h", None):
            load().gcpsl_destroy(self._h)
            self._h = None

    __del__ = close

    @property
    def handle(self):
        return self._h

    def step(self, stats: bool = False):
        """One local round of every cluster; returns (loss[C], active[C])
        when stats is set (one device->host read), else None."""
        _check(load().gcpsl_step(self._h, ct.byref(self._stats) if stats else None), self._h)
        if stats:
            return self._loss.copy(), self._active.copy()
        return None

    def fuse(self):
        _check(load().gcpsl_fuse(self._h), self._h)

    def params(self, cluster: int, segment: int):
        n = self.P_client if segment == GCPSL_CLIENT else self.P_server
        out = np.empty(n, dtype=np.float32)
        _check(load().gcpsl_get_params(self._h, cluster, segment, _p(out, ct.c_float), n, None),
               self._h)
        return out

    def all_params(self, cluster: int):
        return np.concatenate([self.params(cluster, GCPSL_CLIENT),
                               self.params(cluster, GCPSL_SERVER)])

    def set_params(self, cluster: int, blob):
        blob = np.ascontiguousarray(blob, dtype=np.float32)
        _check(load().gcpsl_set_params(self._h, cluster, _p(blob, ct.c_float), blob.size), self._h)

    def bn_state(self, cluster: int):
        """BatchNorm running statistics of one replica (ResNet-18 split)."""
        n = gcpsl_num_params(self.arch, GCPSL_BN_STATE)
        out = np.empty(n, dtype=np.float32)
        _check(load().gcpsl_get_params(self._h, cluster, GCPSL_BN_STATE, _p(out, ct.c_float), n,
                                       None), self._h)
        return out

    def relu_masks(self):
        """[C][B][E] ReLU decisions of the last round (ResNet-18 split)."""
        n = ct.c_size_t(0)
        _check(load().gcpsl_get_relu_masks(self._h, None, 0, ct.byref(n)), self._h)
        out = np.empty(n.value, dtype=np.uint8)
        _check(load().gcpsl_get_relu_masks(self._h, _p(out, ct.c_uint8), n.value, None), self._h)
        return out.reshape(self.C, self.B, -1)

    def set_bn_state(self, cluster: int, v):
        v = np.ascontiguousarray(v, dtype=np.float32)
        _check(load().gcpsl_set_bn_state(self._h, cluster, _p(v, ct.c_float), v.size), self._h)

    def momentum(self, cluster: int):
        n = self.P_client + self.P_server
        out = np.empty(n, dtype=np.float32)
        _check(load().gcpsl_get_momentum(self._h, cluster, _p(out, ct.c_float), n), self._h)
        return out

    def set_momentum(self, cluster: int, v):
        v = np.ascontiguousarray(v, dtype=np.float32)
        _check(load().gcpsl_set_momentum(self._h, cluster, _p(v, ct.c_float), v.size), self._h)

    def pool_codes(self, layer: int, per_example: int):
        """[C][B][per_example] bytes of conv layer `layer`'s max-pool decisions."""
        n = self.C * self.B * per_example
        out = np.empty(n, dtype=np.uint8)
        _check(load().gcpsl_get_pool_codes(self._h, layer, _p(out, ct.c_uint8), n), self._h)
        return out.reshape(self.C, self.B, per_example)

    def cut(self, which: int):
        n = int(load().gcpsl_cut_elems(self._h))
        out = np.empty(n, dtype=np.float32)
        _check(load().gcpsl_get_cut(self._h, which, _p(out, ct.c_float), n), self._h)
        return out.reshape(self.C, self.B, -1)

    def sample(self):
        idx = np.empty((self.C, self.B), dtype=np.int32)
        counts = np.empty((self.C, self.K), dtype=np.int32)
        _check(load().gcpsl_get_sample(self._h, _p(idx, ct.c_int32), _p(counts, ct.c_int32)),
               self._h)
        return idx, counts

    @property
    def rounds(self) -> int:
        return int(load().gcpsl_rounds(self._h))

    def set_stream(self, stream_ptr: int | None):
        _check(load().gcpsl_set_stream(self._h, ct.c_void_p(stream_ptr) if stream_ptr else None),
               self._h)

    def set_timing(self, on: bool):
        _check(load().gcpsl_set_timing(self._h, int(on)), self._h)

    def kernels_launched(self) -> int:
        """Kernels launched so far (eager launches and graph kernel nodes)."""
        return int(load().gcpsl_kernels_launched(self._h))

    def set_timing_filter(self, prefix=None):
        """Time only kernels whose name starts with prefix (None: all)."""
        _check(load().gcpsl_set_timing_filter(self._h, prefix.encode() if prefix else None),
               self._h)

    def check_wait_timeout(self, limit_ns: int):
        """Runs the bounded-wait failure path (see gcpsl.h); raises the
        resulting GcpslError (GCPSL_E_TIMEOUT)."""
        _check(load().gcpsl_check_wait_timeout(self._h, int(limit_ns)), self._h)

    def set_graph(self, on: bool):
        """Replay rounds from CUDA graphs (default) or launch them eagerly."""
        _check(load().gcpsl_set_graph(self._h, int(on)), self._h)

    def kernel_times(self):
        """{kernel kind: (launches, total device ms)} since the last reset."""
        cap = 64
        names = (ct.c_char_p * cap)()
        launches = (ct.c_int64 * cap)()
        ms = (ct.c_double * cap)()
        n = load().gcpsl_kernel_times(self._h, names, launches, ms, cap)
        return {names[i].decode(): (int(launches[i]), float(ms[i])) for i in range(min(n, cap))}

    def reset_kernel_times(self):
        load().gcpsl_reset_kernel_times(self._h)
