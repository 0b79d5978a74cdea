"""Thin Python binding of libpnn.so (include/pnn.h).

Argument marshalling only: every step of the training path runs in the
library's CUDA kernels.  PyTorch provides the device workspace and streams.
If the library has not been built this module raises; there is no fallback.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libpnn.so")

PNN_OK = 0
PRECISION = {"bf16": 0, "fp32": 1}
CORRECTION = {"residual": 0, "delta": 1}
LAYER_OP = {"conv": 0, "conv_bn_relu": 1, "basic": 2, "bottleneck": 3, "coarse_ru": 4}
HEAD = {"gap_fc": 0, "bn_relu_gap_fc": 1, "gap_mlp": 2}
CJ_POST = {"none": 0, "bn_relu": 1}
TENSOR = {"x": 0, "y": 1, "r": 2, "rtilde": 3, "ytilde": 4, "D": 5, "logits": 6}


class PnnError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"pnn status {status}: {msg}")
        self.status = status


class Layer(C.Structure):
    _fields_ = [("op", C.c_int32), ("cout", C.c_int32), ("mid", C.c_int32), ("k", C.c_int32),
                ("stride", C.c_int32), ("pool", C.c_int32)]


class Desc(C.Structure):
    _fields_ = [("batch", C.c_int32), ("in_c", C.c_int32), ("in_h", C.c_int32), ("in_w", C.c_int32),
                ("classes", C.c_int32),
                ("stem", C.POINTER(Layer)), ("n_stem", C.c_int32),
                ("body", C.POINTER(Layer)), ("n_body", C.c_int32),
                ("segments", C.POINTER(C.c_int32)), ("n_seg", C.c_int32),
                ("coarse", C.POINTER(Layer)), ("coarse_len", C.POINTER(C.c_int32)),
                ("cj_post", C.c_int32), ("head_kind", C.c_int32),
                ("head_hidden", C.POINTER(C.c_int32)), ("n_hidden", C.c_int32)]


class Options(C.Structure):
    _fields_ = [("precision", C.c_int32), ("correction", C.c_int32), ("seed", C.c_uint64),
                ("lr", C.c_float), ("momentum", C.c_float), ("weight_decay", C.c_float),
                ("nesterov", C.c_int32), ("stream_fp32", C.c_int32), ("conv_impl", C.c_int32),
                ("grad_fp32", C.c_int32),
                ("stream", C.c_void_p), ("bn_momentum", C.c_float), ("inference", C.c_int32),
                ("overlap", C.c_int32), ("fuse_correction", C.c_int32)]


class ConvArgs(C.Structure):
    _fields_ = [("batch", C.c_int32), ("h", C.c_int32), ("w", C.c_int32), ("c", C.c_int32),
                ("k", C.c_int32), ("ksize", C.c_int32), ("stride", C.c_int32),
                ("x", C.c_void_p), ("x_dtype", C.c_int32),
                ("bn_scale", C.c_void_p), ("bn_shift", C.c_void_p), ("relu", C.c_int32),
                ("wt", C.c_void_p), ("y", C.c_void_p), ("y_dtype", C.c_int32),
                ("res", C.c_void_p), ("res_dtype", C.c_int32),
                ("y_mean", C.c_void_p), ("y_rstd", C.c_void_p),
                ("dy", C.c_void_p), ("dx", C.c_void_p), ("accumulate", C.c_int32),
                ("bn_mean", C.c_void_p), ("bn_rstd", C.c_void_p), ("dgamma", C.c_void_p), ("dbeta", C.c_void_p),
                ("dw", C.c_void_p)]


class Trace(C.Structure):
    _fields_ = [("kind", C.c_int32), ("variant", C.c_int32), ("phase", C.c_int32), ("instances", C.c_int32),
                ("tiles", C.c_int32),
                ("shape", C.c_int32 * 6), ("block", C.c_int32), ("ms", C.c_double), ("flops", C.c_double),
                ("bytes", C.c_double)]


_lib = None


def load():
    """Load libpnn.so; raises if it is missing (run build() first)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built; call __graft_entry__.build() or "
                          "paper_2103_08802_gb300.build.build()")
    lib = C.CDLL(LIB_PATH)
    P, I32, SZ = C.c_void_p, C.c_int32, C.c_size_t
    sig = {
        "pnn_default_options": (None, [C.POINTER(Options)]),
        "pnn_create": (C.c_int, [C.POINTER(Desc), C.POINTER(Options), C.POINTER(P)]),
        "pnn_workspace_bytes": (C.c_int, [P, C.POINTER(SZ)]),
        "pnn_bind_workspace": (C.c_int, [P, P, SZ]),
        "pnn_forward": (C.c_int, [P, P, P, P]),
        "pnn_backward": (C.c_int, [P]),
        "pnn_sgd_step": (C.c_int, [P, C.c_float]),
        "pnn_train_step": (C.c_int, [P, P, P, P]),
        "pnn_train_step_host": (C.c_int, [P, P, P, P]),
        "pnn_sync": (C.c_int, [P]),
        "pnn_destroy": (None, [P]),
        "pnn_num_params": (C.c_int, [P, C.POINTER(SZ)]),
        "pnn_num_param_tensors": (C.c_int, [P, C.POINTER(I32)]),
        "pnn_param_tensor_info": (C.c_int, [P, I32, C.POINTER(I32), C.POINTER(I32), C.POINTER(SZ)]),
        "pnn_get_params": (C.c_int, [P, P, SZ]),
        "pnn_set_params": (C.c_int, [P, P, SZ]),
        "pnn_get_grads": (C.c_int, [P, P, SZ]),
        "pnn_get_momentum": (C.c_int, [P, P, SZ]),
        "pnn_tensor_size": (C.c_int, [P, I32, I32, C.POINTER(SZ)]),
        "pnn_get_tensor": (C.c_int, [P, I32, I32, P, SZ]),
        "pnn_get_timings": (C.c_int, [P, C.POINTER(C.c_float)]),
        "pnn_time_phases": (C.c_int, [P, C.c_void_p, C.c_void_p, C.c_int32, C.POINTER(C.c_float)]),
        "pnn_block_costs": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.POINTER(C.c_double), C.c_int32]),
        "pnn_running_stats_size": (C.c_int, [P, C.POINTER(C.c_size_t)]),
        "pnn_get_running_stats": (C.c_int, [P, C.c_void_p, C.c_size_t]),
        "pnn_set_running_stats": (C.c_int, [P, C.c_void_p, C.c_size_t]),
        "pnn_infer": (C.c_int, [P, C.c_void_p, C.c_void_p]),
        "pnn_partition": (C.c_int, [C.POINTER(C.c_double), C.c_int32, C.c_int32, C.POINTER(C.c_int32)]),
        "pnn_launch_counts": (C.c_int, [P, C.POINTER(I32)]),
        "pnn_profile": (C.c_int, [P, I32]),
        "pnn_profile_read": (C.c_int, [P, I32, C.POINTER(C.c_double), C.POINTER(C.c_int64),
                                       C.POINTER(C.c_double), C.POINTER(C.c_double)]),
        "pnn_profile_trace": (C.c_int, [P, I32, C.POINTER(Trace), C.POINTER(I32)]),
        "pnn_num_kernel_kinds": (I32, []),
        "pnn_debug_word": (C.c_uint64, []),
        "pnn_kernel_kind_name": (C.c_char_p, [I32]),
        "pnn_conv_wgrad_noalloc": (C.c_int, [P, P, P, I32, I32, I32, I32, I32, I32, I32, P]),
        "pnn_selftest_wait_timeout": (C.c_int, [C.c_int64, P]),
        "pnn_conv_workspace_bytes": (C.c_int, [I32, I32, I32, C.POINTER(ConvArgs), C.POINTER(SZ)]),
        "pnn_conv_run": (C.c_int, [I32, I32, I32, C.POINTER(ConvArgs), P, SZ, P]),
        "pnn_conv_time": (C.c_int, [I32, I32, I32, C.POINTER(ConvArgs), P, SZ, P, I32, C.POINTER(C.c_float)]),
        "pnn_last_error": (C.c_char_p, [P]),
        "pnn_status_string": (C.c_char_p, [C.c_int]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _layers(specs):
    arr = (Layer * max(1, len(specs)))()
    for i, s in enumerate(specs):
        arr[i] = Layer(LAYER_OP[s["op"]], s["cout"], s.get("mid", 0), s.get("k", 3), s.get("stride", 1),
                       s.get("pool", 0))
    return arr


def _make_desc(desc):
    """The C description of a description dict, and the arrays it points to."""
    d = Desc()
    d.batch, d.in_c, d.in_h, d.in_w = desc["batch"], desc["in_c"], desc["in_h"], desc["in_w"]
    d.classes = desc["classes"]
    stem, body = _layers(desc["stem"]), _layers(desc["body"])
    segs = (C.c_int32 * len(desc["segments"]))(*desc["segments"])
    flat = [l for F in desc["coarse"] for l in F]
    coarse = _layers(flat)
    clen = (C.c_int32 * max(1, len(desc["coarse"])))(*[len(F) for F in desc["coarse"]])
    hidden = list(desc["head"].get("hidden", []))
    hid = (C.c_int32 * max(1, len(hidden)))(*hidden)
    d.stem, d.n_stem = stem, len(desc["stem"])
    d.body, d.n_body = body, len(desc["body"])
    d.segments, d.n_seg = segs, len(desc["segments"])
    d.coarse, d.coarse_len = coarse, clen
    d.cj_post = CJ_POST[desc["cj_post"]]
    d.head_kind = HEAD[desc["head"]["kind"]]
    d.head_hidden, d.n_hidden = hid, len(hidden)
    return d, [stem, body, segs, coarse, clen, hid]


def _global_check(lib, status):
    if status != PNN_OK:
        msg = lib.pnn_last_error(None)
        raise PnnError(status, msg.decode() if msg else "")


COST = {"flops": 0, "bytes": 1}


def block_costs(desc, kind="flops"):
    """Per-layer cost of the body (forward + backward of the untorn network):
    a list of len(desc["body"]) floats.  Host only."""
    lib = load()
    d, keep = _make_desc(desc)
    o = Options()
    lib.pnn_default_options(C.byref(o))
    o.precision = PRECISION[desc["precision"]]
    n = len(desc["body"])
    out = (C.c_double * n)()
    _global_check(lib, lib.pnn_block_costs(C.byref(d), C.byref(o), COST[kind], out, n))
    return list(out)


def partition(costs, n_seg):
    """Layers per segment of the min-max contiguous cut of `costs`.  Host only."""
    lib = load()
    n = len(costs)
    c = (C.c_double * max(1, n))(*costs)
    seg = (C.c_int32 * max(1, n_seg))()
    _global_check(lib, lib.pnn_partition(c, n, n_seg, seg))
    return list(seg)[:n_seg]


def balanced_segments(desc, n_seg, kind="flops"):
    """Segments of `desc`'s body of equal cost (Section 4.2's remark)."""
    return partition(block_costs(desc, kind), n_seg)


class ParaNet:
    """A parareal network planned and trained by libpnn.

    desc: a description dict (see workloads).  The workspace is one torch
    uint8 tensor on `device`."""

    def __init__(self, desc, precision=None, correction=None, seed=0, lr=0.1, momentum=0.9,
                 weight_decay=5e-4, nesterov=True, stream_fp32=None, conv_impl=0, grad_fp32=False, stream=None,
                 device="cuda", bind=True, inference=False, bn_momentum=0.1, overlap=0, fuse_correction=True):
        self.lib = load()
        self.desc = desc
        d, self._keep = _make_desc(desc)
        o = Options()
        self.lib.pnn_default_options(C.byref(o))
        o.precision = PRECISION[precision or desc["precision"]]
        o.correction = CORRECTION[correction or desc.get("correction", "residual")]
        o.seed, o.lr, o.momentum, o.weight_decay = seed, lr, momentum, weight_decay
        if stream_fp32 is None:  # the description's storage of the residual stream (fp32 if unstated)
            stream_fp32 = desc.get("residual_stream", "fp32") == "fp32"
        o.nesterov, o.stream_fp32, o.conv_impl = int(nesterov), int(stream_fp32), int(conv_impl)
        o.grad_fp32 = int(grad_fp32)
        o.inference, o.bn_momentum, o.overlap = int(inference), bn_momentum, int(overlap)
        o.fuse_correction = int(fuse_correction)
        self.stream = stream
        o.stream = None if stream is None else C.c_void_p(stream.cuda_stream)
        self.h = C.c_void_p()
        self._check(self.lib.pnn_create(C.byref(d), C.byref(o), C.byref(self.h)), global_err=True)
        sz = C.c_size_t()
        self._check(self.lib.pnn_workspace_bytes(self.h, C.byref(sz)))
        self.workspace_bytes = sz.value
        self.device = device
        self.ws = None
        if bind:
            self.bind()

    # ------------------------------------------------------------ plumbing
    def _check(self, status, global_err=False):
        if status != PNN_OK:
            msg = self.lib.pnn_last_error(None if global_err else self.h)
            raise PnnError(status, msg.decode() if msg else "")

    def bind(self):
        import torch
        self.ws = torch.empty(self.workspace_bytes, dtype=torch.uint8, device=self.device)
        self._check(self.lib.pnn_bind_workspace(self.h, C.c_void_p(self.ws.data_ptr()), self.workspace_bytes))

    def close(self):
        if getattr(self, "h", None):
            self.lib.pnn_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ------------------------------------------------------------ step
    def _args(self, x, labels, loss):
        import torch
        d = self.desc
        if x.dtype != torch.float32 or not x.is_cuda or not x.is_contiguous() \
                or tuple(x.shape) != (d["batch"], d["in_c"], d["in_h"], d["in_w"]):
            raise TypeError("x must be a contiguous float32 CUDA tensor of shape (batch, C, H, W)")
        if labels.dtype != torch.int32 or not labels.is_cuda or labels.numel() != d["batch"]:
            raise TypeError("labels must be an int32 CUDA tensor of length batch")
        if loss is not None and (loss.dtype != torch.float32 or not loss.is_cuda):
            raise TypeError("loss must be a float32 CUDA tensor")

    def forward(self, x, labels, loss=None):
        self._args(x, labels, loss)
        self._check(self.lib.pnn_forward(self.h, C.c_void_p(x.data_ptr()), C.c_void_p(labels.data_ptr()),
                                         None if loss is None else C.c_void_p(loss.data_ptr())))

    def backward(self):
        self._check(self.lib.pnn_backward(self.h))

    def sgd_step(self, lr=0.0):
        self._check(self.lib.pnn_sgd_step(self.h, lr))

    def train_step(self, x, labels, loss=None):
        self._args(x, labels, loss)
        self._check(self.lib.pnn_train_step(self.h, C.c_void_p(x.data_ptr()), C.c_void_p(labels.data_ptr()),
                                            None if loss is None else C.c_void_p(loss.data_ptr())))

    def train_step_host(self, x, labels):
        """x: float32 NCHW host array (ideally pinned), labels int32."""
        out = C.c_float()
        xp = x.data_ptr() if hasattr(x, "data_ptr") else x.ctypes.data
        lp = labels.data_ptr() if hasattr(labels, "data_ptr") else labels.ctypes.data
        self._check(self.lib.pnn_train_step_host(self.h, C.c_void_p(xp), C.c_void_p(lp), C.byref(out)))
        return out.value

    def sync(self):
        self._check(self.lib.pnn_sync(self.h))

    # ------------------------------------------------------------ parameters
    @property
    def num_params(self):
        n = C.c_size_t()
        self._check(self.lib.pnn_num_params(self.h, C.byref(n)))
        return n.value

    def param_spec(self):
        """[(kind, dims, offset)] in theta-bar order."""
        n = C.c_int32()
        self._check(self.lib.pnn_num_param_tensors(self.h, C.byref(n)))
        out = []
        for i in range(n.value):
            k, dims, off = C.c_int32(), (C.c_int32 * 4)(), C.c_size_t()
            self._check(self.lib.pnn_param_tensor_info(self.h, i, C.byref(k), dims, C.byref(off)))
            out.append((k.value, tuple(dims), off.value))
        return out

    def _vec(self, fn):
        a = np.empty(self.num_params, dtype=np.float32)
        self._check(fn(self.h, C.c_void_p(a.ctypes.data), a.size))
        return a

    def get_params(self):
        return self._vec(self.lib.pnn_get_params)

    def get_grads(self):
        return self._vec(self.lib.pnn_get_grads)

    def get_momentum(self):
        return self._vec(self.lib.pnn_get_momentum)

    def set_params(self, theta):
        a = np.ascontiguousarray(theta, dtype=np.float32)
        self._check(self.lib.pnn_set_params(self.h, C.c_void_p(a.ctypes.data), a.size))

    # ------------------------------------------------------------ tensors
    def tensor_size(self, which, j=0):
        n = C.c_size_t()
        self._check(self.lib.pnn_tensor_size(self.h, TENSOR[which], j, C.byref(n)))
        return n.value

    def get_tensor(self, which, j=0):
        n = self.tensor_size(which, j)
        if n == 0:
            raise KeyError((which, j))
        a = np.empty(n, dtype=np.float32)
        self._check(self.lib.pnn_get_tensor(self.h, TENSOR[which], j, C.c_void_p(a.ctypes.data), n))
        return a

    def timings(self):
        ms = (C.c_float * 10)()
        self._check(self.lib.pnn_get_timings(self.h, ms))
        keys = ["pre_f", "fine_f", "coarse_f", "post_f", "pre_b", "fine_b", "coarse_b", "post_b", "update", "total"]
        return dict(zip(keys, list(ms)))

    def running_stats(self):
        """BN running statistics (per BN layer in parameter order: C means, C variances)."""
        n = C.c_size_t()
        self._check(self.lib.pnn_running_stats_size(self.h, C.byref(n)))
        a = np.empty(n.value, dtype=np.float32)
        self._check(self.lib.pnn_get_running_stats(self.h, C.c_void_p(a.ctypes.data), n.value))
        return a

    def set_running_stats(self, a):
        a = np.ascontiguousarray(a, dtype=np.float32)
        self._check(self.lib.pnn_set_running_stats(self.h, C.c_void_p(a.ctypes.data), a.size))

    def infer(self, x, logits):
        """Eval-mode forward of an inference net: x (device NCHW float32) ->
        logits (device float32 batch x classes), asynchronous on the stream."""
        import torch
        d = self.desc
        if x.dtype != torch.float32 or not x.is_cuda or not x.is_contiguous() \
                or tuple(x.shape) != (d["batch"], d["in_c"], d["in_h"], d["in_w"]):
            raise TypeError("x must be a contiguous float32 CUDA tensor of shape (batch, C, H, W)")
        if logits.dtype != torch.float32 or not logits.is_cuda or not logits.is_contiguous() \
                or logits.numel() != d["batch"] * d["classes"]:
            raise TypeError("logits must be a contiguous float32 CUDA tensor of batch x classes")
        self._check(self.lib.pnn_infer(self.h, C.c_void_p(x.data_ptr()), C.c_void_p(logits.data_ptr())))

    def time_phases(self, x, labels, steps=5):
        """Per-phase ms of `steps` graph-replayed training steps (device x, labels)."""
        self._args(x, labels, None)
        ms = (C.c_float * 10)()
        self._check(self.lib.pnn_time_phases(self.h, C.c_void_p(x.data_ptr()), C.c_void_p(labels.data_ptr()),
                                             int(steps), ms))
        keys = ["pre_f", "fine_f", "coarse_f", "post_f", "pre_b", "fine_b", "coarse_b", "post_b", "update", "total"]
        return dict(zip(keys, list(ms)))

    def profile(self, enable=True):
        self._check(self.lib.pnn_profile(self.h, int(enable)))

    def profile_read(self):
        """{kind name: (ms, launches, flops, bytes)} accumulated since profile()."""
        out = {}
        for k in range(self.lib.pnn_num_kernel_kinds()):
            ms, n, fl, by = C.c_double(), C.c_int64(), C.c_double(), C.c_double()
            self._check(self.lib.pnn_profile_read(self.h, k, C.byref(ms), C.byref(n), C.byref(fl), C.byref(by)))
            if n.value:
                out[self.lib.pnn_kernel_kind_name(k).decode()] = (ms.value, n.value, fl.value, by.value)
        return out

    def profile_trace(self):
        """Per-launch records since profile(): list of dicts in launch order."""
        n = C.c_int32()
        self._check(self.lib.pnn_profile_trace(self.h, 0, None, C.byref(n)))
        buf = (Trace * max(1, n.value))()
        self._check(self.lib.pnn_profile_trace(self.h, n.value, buf, C.byref(n)))
        return [{"kind": self.lib.pnn_kernel_kind_name(r.kind).decode(), "variant": r.variant, "phase": r.phase,
                 "instances": r.instances, "tiles": r.tiles, "shape": tuple(r.shape), "block": r.block,
                 "ms": r.ms, "flops": r.flops, "bytes": r.bytes} for r in buf[:n.value]]

    def launch_counts(self):
        c = (C.c_int32 * 3)()
        self._check(self.lib.pnn_launch_counts(self.h, c))
        return list(c)


CONV_MODE = {"forward": 0, "dgrad": 1, "wgrad": 2}
CONV_IMPL = {"auto": 0, "tma": 1, "gathered": 2, "tma_tap": 3}
DTYPE = {"f32": 0, "bf16": 1}


def _ptr(t):
    return None if t is None else t.data_ptr()


def _dt(t):
    import torch
    return DTYPE["bf16"] if t is not None and t.dtype == torch.bfloat16 else DTYPE["f32"]


def conv_run(mode, instances, impl="auto", stream=None, repeat=0):
    """One grouped convolution (pnn_conv_run) over `instances`, a list of dicts
    with the geometry (batch, h, w, c, k, ksize, stride) and torch CUDA tensors
    by the names of pnn_conv_args (x, bn_scale, bn_shift, relu, wt, y, res,
    y_mean, y_rstd, dy, dx, accumulate, bn_mean, bn_rstd, dgamma, dbeta, dw).
    The workspace comes from torch.  With repeat > 0 the kernel runs that many
    more times between CUDA events (pnn_conv_time) and the mean device ms of
    one launch is returned.  Raises PnnError on failure."""
    import torch
    lib = load()
    n = len(instances)
    arr = (ConvArgs * n)()
    for i, g in enumerate(instances):
        a = arr[i]
        for key in ("batch", "h", "w", "c", "k", "ksize", "stride"):
            setattr(a, key, int(g[key]))
        a.relu = int(g.get("relu", 0))
        a.accumulate = int(g.get("accumulate", 0))
        for key in ("x", "bn_scale", "bn_shift", "wt", "y", "res", "y_mean", "y_rstd", "dy", "dx", "bn_mean",
                    "bn_rstd", "dgamma", "dbeta", "dw"):
            setattr(a, key, _ptr(g.get(key)))
        a.x_dtype, a.y_dtype, a.res_dtype = _dt(g.get("x")), _dt(g.get("y")), _dt(g.get("res"))
    m, im = CONV_MODE[mode], CONV_IMPL[impl]
    nb = C.c_size_t()
    _global_check(lib, lib.pnn_conv_workspace_bytes(m, im, n, arr, C.byref(nb)))
    ws = torch.empty(max(256, nb.value), dtype=torch.uint8, device="cuda")
    st = stream.cuda_stream if stream is not None else None
    if repeat > 0:
        ms = C.c_float()
        _global_check(lib, lib.pnn_conv_time(m, im, n, arr, ws.data_ptr(), ws.numel(), st, repeat, C.byref(ms)))
        return ms.value
    _global_check(lib, lib.pnn_conv_run(m, im, n, arr, ws.data_ptr(), ws.numel(), st))
    return None
