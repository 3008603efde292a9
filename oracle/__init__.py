"""ctypes wrapper of the CPU oracle (``gcpsl_oracle.c``, ``gcpsl_resnet.c``).

TEST INFRASTRUCTURE ONLY: imported by the tests, the smoke check and the CPU
baseline leg of the benchmark, never by the product package.  The oracle is a
plain fp64 restatement of one GCPSL local round and of fusion; see the C
file's header for what it computes and which passages it follows.
"""
from __future__ import annotations

import ctypes as ct
import os
import subprocess
from pathlib import Path

import numpy as np

HERE = Path(__file__).resolve().parent
LIBDIR = HERE / "lib"
LIB = LIBDIR / "libgcpsl_oracle.so"
SRCS = [HERE / "gcpsl_oracle.c", HERE / "gcpsl_resnet.c"]


def build(force: bool = False) -> Path:
    """Compile the oracle with gcc (OpenMP when available)."""
    if LIB.exists() and not force and all(LIB.stat().st_mtime >= s.stat().st_mtime for s in SRCS):
        return LIB
    LIBDIR.mkdir(exist_ok=True)
    tmp = LIBDIR / f".tmp_{os.getpid()}.so"
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared"] + [str(s) for s in SRCS] + [
        "-o", str(tmp), "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, LIB)
    return LIB


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = ct.CDLL(str(build()))
        _declare(_lib)
    return _lib


def _p(t):
    return ct.POINTER(t)


def _declare(L):
    u32p, i32p, f64p, f32p = _p(ct.c_uint32), _p(ct.c_int32), _p(ct.c_double), _p(ct.c_float)
    L.orc_philox4x32_10.argtypes = [u32p, u32p, u32p]
    L.orc_epoch_perm.argtypes = [i32p, ct.c_int64, ct.c_uint32, ct.c_uint32, ct.c_uint64, i32p]
    L.orc_sample_round.argtypes = [i32p, ct.c_int64, ct.c_int, i32p, ct.c_int, i32p, i32p]
    L.orc_sample_round.restype = ct.c_int
    L.orc_num_params.argtypes = [ct.c_int, ct.c_int]
    L.orc_num_params.restype = ct.c_int64
    L.orc_forward_backward.argtypes = [ct.c_int, ct.c_int, ct.c_double, f64p, ct.c_int, f64p, i32p,
                                       f64p, f64p, f64p, f64p, f64p]
    L.orc_fuse_arrays.argtypes = [ct.c_int, ct.c_int64, f64p, f64p, f64p]
    L.orc_init.argtypes = [ct.c_int, ct.c_int, ct.c_double, ct.c_double, ct.c_double, ct.c_int,
                           ct.c_double, ct.c_int, ct.c_int, i32p, ct.c_int, ct.c_int, ct.c_uint64,
                           ct.c_int, f32p, i32p, i32p, ct.c_int64, f32p, _p(ct.c_void_p)]
    L.orc_destroy.argtypes = [ct.c_void_p]
    L.orc_augment_params.argtypes = [ct.c_uint64, ct.c_uint32, ct.c_uint32, ct.c_uint32, i32p]
    L.orc_augment_params.restype = None
    L.orc_augment_image.argtypes = [f32p, ct.c_int, ct.c_int, ct.c_int, f64p]
    L.orc_augment_image.restype = None
    L.orc_set_augment.argtypes = [ct.c_void_p, ct.c_int]
    L.orc_set_augment.restype = None
    L.orc_step.argtypes = [ct.c_void_p]
    L.orc_fuse.argtypes = [ct.c_void_p]
    L.orc_get_params.argtypes = [ct.c_void_p, ct.c_int, ct.c_int, f64p]
    L.orc_set_params.argtypes = [ct.c_void_p, ct.c_int, f64p]
    L.orc_get_sample.argtypes = [ct.c_void_p, i32p, i32p]
    L.orc_get_stats.argtypes = [ct.c_void_p, f64p, i32p]
    L.orc_get_cut.argtypes = [ct.c_void_p, ct.c_int, f64p]
    L.orc_get_cut.restype = ct.c_int64
    L.orc_get_q.argtypes = [ct.c_void_p, f64p]
    L.orc_rounds.argtypes = [ct.c_void_p]
    L.orc_rounds.restype = ct.c_int64
    L.orc_get_momentum.argtypes = [ct.c_void_p, ct.c_int, f64p]
    L.orc_set_momentum.argtypes = [ct.c_void_p, ct.c_int, f64p]
    L.orc_set_tie_tol.argtypes = [ct.c_void_p, ct.c_double]
    L.orc_set_tie_tol.restype = None
    L.orc_get_pool_cand.argtypes = [ct.c_void_p, ct.c_int, _p(ct.c_uint8)]
    L.orc_get_pool_cand.restype = ct.c_int64
    L.orc_get_ties.argtypes = [ct.c_void_p, i32p]
    L.orc_get_ties.restype = None
    L.orc_set_bn_state.argtypes = [ct.c_void_p, ct.c_int, f64p]
    L.orn_forward_backward.argtypes = [ct.c_int, ct.c_int, ct.c_double, f64p, f64p, ct.c_int, f64p, i32p,
                                       f64p, f64p, f64p, f64p, f64p]
    L.orn_forward_backward_masks.argtypes = [ct.c_int, ct.c_int, ct.c_double, f64p, f64p, ct.c_int, f64p,
                                             i32p, f64p, f64p, f64p, f64p, f64p,
                                             _p(ct.c_uint8), _p(ct.c_uint8), f64p]
    L.orn_mask_elems.restype = ct.c_int64
    L.orn_set_relu_tol.argtypes = [ct.c_double]
    L.orn_set_relu_tol.restype = None
    L.orc_set_relu_masks.argtypes = [ct.c_void_p, _p(ct.c_uint8)]
    L.orc_get_relu_masks.argtypes = [ct.c_void_p, _p(ct.c_uint8)]
    L.orn_set_norm.argtypes = [ct.c_int, ct.c_double, ct.c_double]
    L.orc_set_norm.argtypes = [ct.c_void_p, ct.c_int, ct.c_double, ct.c_double]
    L.orc_set_client_average.argtypes = [ct.c_void_p, ct.c_int]
    L.orn_init_bn_state.argtypes = [f64p]
    L.orn_init_bn_state.restype = None
    L.orc_set_threads.argtypes = [ct.c_int]
    L.orc_get_threads.restype = ct.c_int


def _ptr(a, t):
    return a.ctypes.data_as(ct.POINTER(t))


def philox4x32_10(ctr, key):
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    o = np.zeros(4, dtype=np.uint32)
    lib().orc_philox4x32_10(_ptr(c, ct.c_uint32), _ptr(k, ct.c_uint32), _ptr(o, ct.c_uint32))
    return o


def epoch_perm(ids, cluster: int, epoch: int, seed: int):
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    out = np.empty_like(ids)
    lib().orc_epoch_perm(_ptr(ids, ct.c_int32), ids.size, cluster, epoch, seed, _ptr(out, ct.c_int32))
    return out


def sample_round(perm, s: int, B: int, owner, K: int):
    perm = np.ascontiguousarray(perm, dtype=np.int32)
    owner = np.ascontiguousarray(owner, dtype=np.int32)
    idx = np.empty(B, dtype=np.int32)
    counts = np.empty(K, dtype=np.int32)
    act = lib().orc_sample_round(_ptr(perm, ct.c_int32), s, B, _ptr(owner, ct.c_int32), K,
                                 _ptr(idx, ct.c_int32), _ptr(counts, ct.c_int32))
    return idx, counts, act


def augment_params(seed: int, t: int, cluster: int, pos: int):
    """(dy, dx, flip) of the sampled image at batch position `pos` of
    cluster `cluster` in round `t` (Section V-A crop + flip; Philox draw)."""
    out = np.zeros(3, dtype=np.int32)
    lib().orc_augment_params(seed, t, cluster, pos, _ptr(out, ct.c_int32))
    return int(out[0]), int(out[1]), int(out[2])


def augment_image(img, dy: int, dx: int, flip: int):
    """The crop at (dy, dx) of the 4-pixel zero-padded CHW image, mirrored
    when flip (fp64)."""
    src = np.ascontiguousarray(img, dtype=np.float32).reshape(3, 32, 32)
    out = np.zeros((3, 32, 32))
    lib().orc_augment_image(_ptr(src, ct.c_float), dy, dx, flip, _ptr(out, ct.c_double))
    return out


def num_params(arch: int, segment: int) -> int:
    return int(lib().orc_num_params(arch, segment))


RESNET18 = 2
RESNET18_C100 = 3          # the same split with a 100-class head


def bn_state_size() -> int:
    """BatchNorm running statistics per replica of the ResNet-18 split."""
    return num_params(RESNET18, 2)


def initial_bn_state():
    out = np.zeros(bn_state_size())
    lib().orn_init_bn_state(_ptr(out, ct.c_double))
    return out


def set_relu_tol(tol: float):
    """Width, in units of a layer's RMS pre-ReLU value, under which a ReLU
    decision is recorded as ambiguous (ResNet-18 split)."""
    lib().orn_set_relu_tol(tol)


def resnet_mask_elems() -> int:
    """ReLU decisions per example of the ResNet-18 split (see masks below)."""
    return int(lib().orn_mask_elems())


def resnet_forward_backward(params, x, labels, bn_state=None, bf16: bool = False,
                            label_smoothing: float = 0.0, want_grad: bool = True,
                            masks_in=None, want_masks: bool = False, classes: int = 10,
                            gn_groups: int = 32, norm_eps: float = 1e-5,
                            bn_momentum: float = 0.1, cut_scale=None):
    """ResNet-18 split with a `classes`-way head (10 or 100): (loss, grad[P]
    or None, cut_act, cut_grad, logits, bn_state after this batch's update of
    the running statistics[, masks]).  masks: [B][resnet_mask_elems()] uint8
    ReLU decisions (stem, then per block those of a1 and of the output, NCHW);
    masks_in replays given decisions.  gn_groups / norm_eps / bn_momentum:
    the norms' hyper-parameters (PyTorch's defaults with 32 groups).
    cut_scale ([B], optional) multiplies each example's gradient at the cut
    before the client backward."""
    params = np.ascontiguousarray(params, dtype=np.float64)
    x = np.ascontiguousarray(x, dtype=np.float64)
    labels = np.ascontiguousarray(labels, dtype=np.int32)
    B = labels.size
    arch = {10: RESNET18, 100: RESNET18_C100}[classes]
    P = num_params(arch, 0) + num_params(arch, 1)
    bn = np.ascontiguousarray(initial_bn_state() if bn_state is None else bn_state,
                              dtype=np.float64).copy()
    loss = np.zeros(1)
    grad = np.zeros(P) if want_grad else None
    ncut = _cut_elems(arch, B)
    ca, cg = np.zeros(ncut), np.zeros(ncut)
    logits = np.zeros(B * classes)
    mo = np.zeros((B, resnet_mask_elems()), dtype=np.uint8) if want_masks else None
    mi = None
    if masks_in is not None:
        mi = np.ascontiguousarray(masks_in, dtype=np.uint8)
        assert mi.size == B * resnet_mask_elems()
    if lib().orn_set_norm(gn_groups, norm_eps, bn_momentum):
        raise ValueError("bad norm hyper-parameters")
    try:
        cs = None if cut_scale is None else np.ascontiguousarray(cut_scale, dtype=np.float64)
        assert cs is None or cs.size == B
        rc = _resnet_pass(classes, bf16, label_smoothing, params, bn, B, x, labels, loss, grad,
                          want_grad, ca, cg, logits, mi, mo, cs)
    finally:
        lib().orn_set_norm(32, 1e-5, 0.1)
    if rc:
        raise RuntimeError(f"oracle resnet forward_backward failed: {rc}")
    out = (float(loss[0]), grad, ca, cg, logits.reshape(B, classes), bn)
    return out + (mo,) if want_masks else out


def _resnet_pass(classes, bf16, label_smoothing, params, bn, B, x, labels, loss, grad, want_grad,
                 ca, cg, logits, mi, mo, cs):
    return lib().orn_forward_backward_masks(
        classes, int(bf16), label_smoothing, _ptr(params, ct.c_double), _ptr(bn, ct.c_double), B,
        _ptr(x, ct.c_double), _ptr(labels, ct.c_int32), _ptr(loss, ct.c_double),
        _ptr(grad, ct.c_double) if want_grad else None, _ptr(ca, ct.c_double),
        _ptr(cg, ct.c_double), _ptr(logits, ct.c_double),
        _ptr(mi, ct.c_uint8) if mi is not None else None,
        _ptr(mo, ct.c_uint8) if mo is not None else None,
        _ptr(cs, ct.c_double) if cs is not None else None)


def forward_backward(arch: int, params, x, labels, bf16: bool = False, label_smoothing: float = 0.0,
                     want_grad: bool = True):
    """(loss, grad[P] or None, cut_act, cut_grad, logits) for one replica."""
    params = np.ascontiguousarray(params, dtype=np.float64)
    x = np.ascontiguousarray(x, dtype=np.float64)
    labels = np.ascontiguousarray(labels, dtype=np.int32)
    B = labels.size
    P = num_params(arch, 0) + num_params(arch, 1)
    loss = np.zeros(1)
    grad = np.zeros(P) if want_grad else None
    ncut = _cut_elems(arch, B)
    ca, cg = np.zeros(ncut), np.zeros(ncut)
    logits = np.zeros(B * 10)
    rc = lib().orc_forward_backward(arch, int(bf16), label_smoothing, _ptr(params, ct.c_double), B,
                                    _ptr(x, ct.c_double), _ptr(labels, ct.c_int32),
                                    _ptr(loss, ct.c_double),
                                    _ptr(grad, ct.c_double) if want_grad else None,
                                    _ptr(ca, ct.c_double), _ptr(cg, ct.c_double),
                                    _ptr(logits, ct.c_double))
    if rc:
        raise RuntimeError(f"oracle forward_backward failed: {rc}")
    return float(loss[0]), grad, ca, cg, logits.reshape(B, 10)


def _cut_elems(arch: int, B: int) -> int:
    return B * {0: 16 * 16 * 16, 1: 64 * 16 * 16, 2: 64 * 32 * 32, 3: 64 * 32 * 32}[arch]


def cut_shape(arch: int):
    return {0: (16, 16, 16), 1: (64, 16, 16), 2: (64, 32, 32), 3: (64, 32, 32)}[arch]


def fuse_arrays(q, theta):
    q = np.ascontiguousarray(q, dtype=np.float64)
    theta = np.ascontiguousarray(theta, dtype=np.float64)
    C, P = theta.shape
    out = np.zeros(P)
    lib().orc_fuse_arrays(C, P, _ptr(q, ct.c_double), _ptr(theta, ct.c_double), _ptr(out, ct.c_double))
    return out


def set_threads(n: int):
    lib().orc_set_threads(n)


def get_threads() -> int:
    return int(lib().orc_get_threads())


class Oracle:
    """C cluster workloads stepped in lockstep by the CPU oracle."""

    def __init__(self, arch, K, C, assignment, B, F, seed, images, labels, owner, init_params,
                 lr=0.05, momentum=0.0, weight_decay=0.0, nesterov=False, label_smoothing=0.0,
                 bf16=False, cluster_base=0, augment=False, gn_groups=32, norm_eps=1e-5,
                 bn_momentum=0.1, client_average=False):
        self.arch, self.K, self.C, self.B = arch, K, C, B
        # the context reads the images in place: keep them alive here
        self._images = np.ascontiguousarray(images, dtype=np.float32)
        self._labels = np.ascontiguousarray(labels, dtype=np.int32)
        self._owner = np.ascontiguousarray(owner, dtype=np.int32)
        self._assign = np.ascontiguousarray(assignment, dtype=np.int32)
        p = np.ascontiguousarray(init_params, dtype=np.float32)
        h = ct.c_void_p()
        rc = lib().orc_init(arch, int(bf16), lr, momentum, weight_decay, int(nesterov),
                            label_smoothing, K, C, _ptr(self._assign, ct.c_int32), B, F, seed,
                            cluster_base, _ptr(self._images, ct.c_float),
                            _ptr(self._labels, ct.c_int32), _ptr(self._owner, ct.c_int32),
                            self._images.shape[0], _ptr(p, ct.c_float), ct.byref(h))
        if rc:
            raise ValueError(f"oracle init failed: {rc}")
        self._h = h
        lib().orc_set_augment(h, int(augment))
        if lib().orc_set_norm(h, gn_groups, norm_eps, bn_momentum):
            self.__del__()
            raise ValueError("bad norm hyper-parameters")
        if lib().orc_set_client_average(h, int(client_average)):
            self.__del__()
            raise MemoryError("oracle allocation failed")
        self.P_client = num_params(arch, 0)
        self.P_server = num_params(arch, 1)

    def __del__(self):
        if getattr(self, "_h", None):
            lib().orc_destroy(self._h)
            self._h = None

    def step(self):
        rc = lib().orc_step(self._h)
        if rc:
            raise RuntimeError(f"oracle step failed: {rc}")

    def fuse(self):
        lib().orc_fuse(self._h)

    def params(self, cluster: int, segment: int):
        n = self.P_client if segment == 0 else self.P_server
        out = np.zeros(n)
        lib().orc_get_params(self._h, cluster, segment, _ptr(out, ct.c_double))
        return out

    def all_params(self, cluster: int):
        return np.concatenate([self.params(cluster, 0), self.params(cluster, 1)])

    def set_params(self, cluster: int, blob):
        blob = np.ascontiguousarray(blob, dtype=np.float64)
        lib().orc_set_params(self._h, cluster, _ptr(blob, ct.c_double))

    def bn_state(self, cluster: int):
        """BatchNorm running statistics of one replica (ResNet-18 split)."""
        out = np.zeros(bn_state_size())
        rc = lib().orc_get_params(self._h, cluster, 2, _ptr(out, ct.c_double))
        if rc:
            raise ValueError("no BatchNorm state for this architecture")
        return out

    def set_bn_state(self, cluster: int, v):
        v = np.ascontiguousarray(v, dtype=np.float64)
        if lib().orc_set_bn_state(self._h, cluster, _ptr(v, ct.c_double)):
            raise ValueError("no BatchNorm state for this architecture")

    def set_relu_masks(self, masks):
        """ResNet-18 split: ReLU decisions ([C][B][resnet_mask_elems()], bit 0)
        that the next round follows instead of its own sign tests."""
        m = np.ascontiguousarray(masks, dtype=np.uint8)
        assert m.size == self.C * self.B * resnet_mask_elems()
        if lib().orc_set_relu_masks(self._h, _ptr(m, ct.c_uint8)):
            raise ValueError("no ReLU records for this architecture")

    def relu_masks(self):
        """[C][B][E] ReLU records of the last round: bit 0 decision used, bit 1
        own sign, bit 2 within the tolerance of 0 (set_relu_tol), bit 3
        within five times it."""
        out = np.zeros((self.C, self.B, resnet_mask_elems()), dtype=np.uint8)
        if lib().orc_get_relu_masks(self._h, _ptr(out, ct.c_uint8)):
            raise ValueError("no ReLU records for this architecture")
        return out

    def momentum(self, cluster: int):
        out = np.zeros(self.P_client + self.P_server)
        lib().orc_get_momentum(self._h, cluster, _ptr(out, ct.c_double))
        return out

    def set_momentum(self, cluster: int, v):
        v = np.ascontiguousarray(v, dtype=np.float64)
        lib().orc_set_momentum(self._h, cluster, _ptr(v, ct.c_double))

    def set_tie_tol(self, tol: float):
        lib().orc_set_tie_tol(self._h, tol)

    def pool_cand(self, layer: int):
        """Per pooled window of the last round, [C][B][cout][Ho][Wo] bytes:
        bits 0-3 valid argmax positions, bit 4 max > 0, bit 5 sign ambiguous
        (None for a layer without pooling)."""
        n = lib().orc_get_pool_cand(self._h, layer, None)
        if n == 0:
            return None
        out = np.zeros(n, dtype=np.uint8)
        lib().orc_get_pool_cand(self._h, layer, _ptr(out, ct.c_uint8))
        return out.reshape(self.C, self.B, -1)

    def ties(self):
        """[C][B] number of ambiguous pooled windows per example, last round."""
        out = np.zeros((self.C, self.B), dtype=np.int32)
        lib().orc_get_ties(self._h, _ptr(out, ct.c_int32))
        return out

    def sample(self):
        idx = np.zeros((self.C, self.B), dtype=np.int32)
        counts = np.zeros((self.C, self.K), dtype=np.int32)
        lib().orc_get_sample(self._h, _ptr(idx, ct.c_int32), _ptr(counts, ct.c_int32))
        return idx, counts

    def stats(self):
        loss = np.zeros(self.C)
        act = np.zeros(self.C, dtype=np.int32)
        lib().orc_get_stats(self._h, _ptr(loss, ct.c_double), _ptr(act, ct.c_int32))
        return loss, act

    def cut(self, which: int):
        n = lib().orc_get_cut(self._h, which, None)
        out = np.zeros(n)
        lib().orc_get_cut(self._h, which, _ptr(out, ct.c_double))
        return out.reshape((self.C, self.B) + cut_shape(self.arch))

    def q(self):
        out = np.zeros(self.C)
        lib().orc_get_q(self._h, _ptr(out, ct.c_double))
        return out

    @property
    def rounds(self) -> int:
        return int(lib().orc_rounds(self._h))
