"""ctypes binding of ``libpolyq.so`` (the C ABI declared in include/polyq.h).

Argument marshalling only: every step of the layer runs in the library.
PyTorch supplies device memory and the current CUDA stream.  Importing this
module fails loudly when the library has not been built.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libpolyq.so")

POLYQ_OK = 0
POLYQ_EINVAL = -1
POLYQ_ENOMEM = -2
POLYQ_ECUDA = -3
POLYQ_EUNSUPPORTED = -4
POLYQ_ETIMEOUT = -5
MAX_BLOCKS = 5
MAX_GROUP = 8
GROUP = 64
NOALLOC_SCRATCH_BYTES = 1 << 20  # scratch compiled in for linear_gemv_noalloc
ALLOC_WATERFILL = 0
PROXY_SALIENCY = 0
PROXY_QUANT = 1
GPU_QUANTA = {2: 64, 3: 128, 4: 32, 8: 16, 16: 8}
ALLOC_LADDER = 1

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with paper_2607_14618_gb300.build.build_library()")
_lib = C.CDLL(LIB_PATH)


class PolyqError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"[{code}] {msg}")
        self.code = code


class PackOpts(C.Structure):
    _fields_ = [("group_size", C.c_int32), ("palette_mask", C.c_uint32),
                ("alloc_rule", C.c_int32), ("snap_quanta", C.c_int32),
                ("n_threads", C.c_int32), ("forced_bits", C.POINTER(C.c_uint8)),
                ("proxy", C.c_int32), ("act_scaling", C.c_int32), ("quanta", C.c_int32 * 5),
                ("act_sqmean", C.POINTER(C.c_float))]


class Block(C.Structure):
    _fields_ = [("bits", C.c_int32), ("n_ch", C.c_int32), ("pos0", C.c_int32),
                ("seg_off", C.c_int32), ("seg_bytes", C.c_int32), ("grp_off", C.c_int32),
                ("n_grp", C.c_int32)]

    def as_dict(self):
        """The block's fields as a dict."""
        return {f: getattr(self, f) for f, _ in self._fields_}


class Info(C.Structure):
    _fields_ = [("N", C.c_int64), ("K", C.c_int64), ("row_stride", C.c_int64),
                ("n_groups", C.c_int64), ("n_blocks", C.c_int32),
                ("blocks", Block * MAX_BLOCKS), ("budget", C.c_double), ("b_real", C.c_double),
                ("packed_bytes", C.c_int64), ("meta_bytes", C.c_int64),
                ("meta_stride", C.c_int64), ("pad_bytes", C.c_int64), ("alpha", C.c_double * 5),
                ("has_xscale", C.c_int32)]


X_BF16, X_F32, X_RMSNORM, X_SILU_MUL = 0, 1, 2, 3


class GemvInput(C.Structure):
    _fields_ = [("kind", C.c_int32), ("eps", C.c_float), ("a", C.c_void_p), ("b", C.c_void_p),
                ("x_out", C.c_void_p)]


NODE_SOURCE_FIXED, NODE_SOURCE_FREE, NODE_LINEAR, NODE_ELEMENTWISE, NODE_BOUNDARY, \
    NODE_ATTENTION = range(6)


class PlanNode(C.Structure):
    _fields_ = [("kind", C.c_int32), ("n_in", C.c_int32), ("in_", C.c_int32 * 3),
                ("out", C.c_int32), ("perm", C.c_int32)]


class DevLayer(C.Structure):
    _fields_ = [("packed", C.c_void_p), ("meta", C.c_void_p), ("gather", C.c_void_p),
                ("N", C.c_int64), ("K", C.c_int64), ("row_stride", C.c_int64),
                ("n_groups", C.c_int64), ("meta_stride", C.c_int64), ("n_blocks", C.c_int32),
                ("blocks", Block * MAX_BLOCKS), ("xscale", C.c_void_p)]


class GemvPhase(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("layers", C.POINTER(DevLayer) * MAX_GROUP),
                ("in_", GemvInput), ("xs", C.c_void_p * MAX_GROUP),
                ("ys", C.c_void_p * MAX_GROUP), ("residuals", C.c_void_p * MAX_GROUP)]


_P = C.c_void_p
_SIGS = {
    "polyq_last_error": (C.c_char_p, []),
    "polyq_pack_opts_default": (None, [C.POINTER(PackOpts)]),
    "polyq_pack": (C.c_int, [_P, C.c_int64, C.c_int64, _P, C.c_double, C.POINTER(PackOpts),
                             C.POINTER(C.c_void_p)]),
    "polyq_free": (None, [_P]),
    "polyq_layer_info": (C.c_int, [_P, C.POINTER(Info)]),
    "polyq_layer_export": (C.c_int, [_P, _P, _P, C.c_int64, _P, _P, _P]),
    "polyq_layer_xscale": (C.c_int, [_P, _P]),
    "polyq_layer_permute_rows": (C.c_int, [_P, _P]),
    "polyq_permute_merge": (C.c_int, [_P, _P, C.c_int64, _P]),
    "polyq_plan_graph": (C.c_int, [C.POINTER(PlanNode), C.c_int32, _P, C.c_int32,
                                   C.POINTER(C.c_void_p), _P, C.c_int32, _P,
                                   C.POINTER(C.c_int64)]),
    "polyq_dev_layer_fill": (C.c_int, [_P, _P, _P, _P, C.POINTER(DevLayer)]),
    "polyq_gemv_workspace_bytes": (C.c_int, [C.POINTER(DevLayer), C.c_int, C.POINTER(C.c_size_t)]),
    "polyq_linear_gemv": (C.c_int, [C.POINTER(DevLayer), _P, C.c_int, _P, _P, _P, C.c_size_t, _P]),
    "polyq_linear_gemv_noalloc": (C.c_int, [C.POINTER(DevLayer), _P, C.c_int, _P, _P, _P]),
    "polyq_noalloc_status": (C.c_int, [C.POINTER(C.c_int), _P]),
    "polyq_gemv_group_workspace_bytes": (C.c_int, [C.POINTER(C.POINTER(DevLayer)), C.c_int,
                                                   C.c_int, C.POINTER(C.c_size_t)]),
    "polyq_linear_gemv_group": (C.c_int, [C.POINTER(C.POINTER(DevLayer)), C.c_int,
                                          C.POINTER(C.c_void_p), C.c_int,
                                          C.POINTER(C.c_void_p), C.POINTER(C.c_void_p),
                                          _P, C.c_size_t, _P]),
    "polyq_linear_gemv_input": (C.c_int, [C.POINTER(C.POINTER(DevLayer)), C.c_int,
                                          C.POINTER(GemvInput), C.c_int,
                                          C.POINTER(C.c_void_p), C.POINTER(C.c_void_p),
                                          _P, C.c_size_t, _P]),
    "polyq_gemv_chain_create": (C.c_int, [C.POINTER(GemvPhase), C.c_int, C.c_int,
                                          C.POINTER(C.c_void_p)]),
    "polyq_gemv_chain_plan_bytes": (C.c_int, [_P, C.POINTER(C.c_size_t)]),
    "polyq_gemv_chain_workspace_bytes": (C.c_int, [_P, C.POINTER(C.c_size_t)]),
    "polyq_gemv_chain_upload": (C.c_int, [_P, _P, C.c_size_t, _P]),
    "polyq_linear_gemv_chain": (C.c_int, [_P, _P, C.c_size_t, _P]),
    "polyq_gemv_chain_free": (None, [_P]),
    "polyq_workspace_status": (C.c_int, [_P, C.POINTER(C.c_int), _P]),
    "polyq_gemm_workspace_bytes": (C.c_int, [C.POINTER(DevLayer), C.c_int64,
                                             C.POINTER(C.c_size_t)]),
    "polyq_linear_gemm": (C.c_int, [C.POINTER(DevLayer), _P, C.c_int64, _P, _P, C.c_size_t, _P]),
    "polyq_unpack_codes": (C.c_int, [C.POINTER(DevLayer), _P, _P]),
    "polyq_f64_to_f16": (C.c_uint16, [C.c_double]),
}
for _name, (_res, _args) in _SIGS.items():
    _fn = getattr(_lib, _name)
    _fn.restype = _res
    _fn.argtypes = _args


def exported_symbols():
    """Names of the C-ABI entry points this binding expects."""
    return list(_SIGS)


def _check(rc):
    if rc != POLYQ_OK:
        raise PolyqError(rc, _lib.polyq_last_error().decode())


def last_error():
    """The calling thread's last error message from the library."""
    return _lib.polyq_last_error().decode()


def f64_to_f16(v: float) -> int:
    """The library's fp64 -> fp16 round-to-nearest-even, as raw bits (a test aid)."""
    return int(_lib.polyq_f64_to_f16(float(v)))


def permute_merge(producer_basis, consumer_perm):
    """gather[p] = producer_basis^-1[consumer_perm[p]] (merge rule, index side)."""
    b = np.ascontiguousarray(producer_basis, dtype=np.int32)
    c = np.ascontiguousarray(consumer_perm, dtype=np.int32)
    if b.shape != c.shape or b.ndim != 1:
        raise ValueError("shape mismatch")
    out = np.empty_like(c)
    _check(_lib.polyq_permute_merge(b.ctypes.data, c.ctypes.data, c.shape[0], out.ctypes.data))
    return out


def plan_graph(nodes, edge_dims, perms):
    """Section 4.4 planning: ``nodes`` as (kind, input edges, output edge or
    -1, permutation id or -1), ``perms`` the linears' permutations.  Returns
    (labels [n_edges] int32, -1 = natural order, modelled bytes per token)."""
    arr = (PlanNode * len(nodes))()
    for i, (kind, ins, out, perm) in enumerate(nodes):
        arr[i].kind = int(kind)
        arr[i].n_in = len(ins)
        for j, e in enumerate(ins):
            arr[i].in_[j] = int(e)
        arr[i].out = int(out)
        arr[i].perm = int(perm)
    dims = np.ascontiguousarray(edge_dims, dtype=np.int64)
    keep = [np.ascontiguousarray(p, dtype=np.int32) for p in perms]
    ptrs = (C.c_void_p * max(1, len(keep)))(*[k.ctypes.data for k in keep])
    lens = np.array([len(k) for k in keep] or [0], dtype=np.int64)
    labels = np.empty(len(dims), np.int32)
    cost = C.c_int64()
    _check(_lib.polyq_plan_graph(arr, len(nodes), dims.ctypes.data, len(dims), ptrs,
                                 lens.ctypes.data, len(keep), labels.ctypes.data, C.byref(cost)))
    return labels, int(cost.value)


def _palette_mask(palette):
    m = 0
    for b in palette:
        m |= 1 << int(b)
    return m


class HostLayer:
    """A packed layer owned by the library (host memory)."""

    def __init__(self, handle):
        self._h = C.c_void_p(handle)

    @classmethod
    def pack(cls, W, act_absmean=None, budget=3.0, forced_bits=None,
             rule=ALLOC_WATERFILL, palette=(2, 3, 4, 8, 16), n_threads=0,
             proxy=PROXY_SALIENCY, snap_quanta=False, quanta=None, act_scaling=False,
             act_sqmean=None):
        """Allocate, (optionally) snap to quanta and scale, cluster and pack.

        ``quanta`` maps widths 2, 3, 4, 8, 16 to channels per quantum (default
        GPU_QUANTA); ``act_sqmean`` is E[x^2] per channel (default
        act_absmean squared)."""
        W = np.ascontiguousarray(W, dtype=np.float32)
        if W.ndim != 2:
            raise ValueError("W must be [N][K]")
        N, K = W.shape
        opts = PackOpts()
        _lib.polyq_pack_opts_default(C.byref(opts))
        opts.alloc_rule = int(rule)
        opts.palette_mask = _palette_mask(palette)
        opts.n_threads = int(n_threads)
        opts.proxy = int(proxy)
        opts.snap_quanta = 1 if snap_quanta else 0
        opts.act_scaling = 1 if act_scaling else 0
        if quanta is not None:
            for i, b in enumerate((2, 3, 4, 8, 16)):
                opts.quanta[i] = int(quanta[b])
        keep_x2 = None
        if act_sqmean is not None:
            keep_x2 = np.ascontiguousarray(act_sqmean, dtype=np.float32)
            if keep_x2.shape != (W.shape[1],):
                raise ValueError("act_sqmean must be [K]")
            opts.act_sqmean = keep_x2.ctypes.data_as(C.POINTER(C.c_float))
        keep = None
        if forced_bits is not None:
            keep = np.ascontiguousarray(forced_bits, dtype=np.uint8)
            if keep.shape != (K,):
                raise ValueError("forced_bits must be [K]")
            opts.forced_bits = keep.ctypes.data_as(C.POINTER(C.c_uint8))
        a = None
        if act_absmean is not None:
            a = np.ascontiguousarray(act_absmean, dtype=np.float32)
            if a.shape != (K,):
                raise ValueError("act_absmean must be [K]")
        h = C.c_void_p()
        _check(_lib.polyq_pack(W.ctypes.data, N, K, a.ctypes.data if a is not None else None,
                               float(budget), C.byref(opts), C.byref(h)))
        return cls(h.value)

    def __del__(self):
        if getattr(self, "_h", None) and self._h.value:
            _lib.polyq_free(self._h)
            self._h = C.c_void_p()

    def info(self) -> dict:
        """Block table, realised budget, byte counts and Section 3.4 factors of the packed layer."""
        inf = Info()
        _check(_lib.polyq_layer_info(self._h, C.byref(inf)))
        d = {f: getattr(inf, f) for f, _ in Info._fields_ if f != "blocks"}
        d["blocks"] = [inf.blocks[i].as_dict() for i in range(inf.n_blocks)]
        d["alpha"] = {b: inf.alpha[i] for i, b in enumerate((2, 3, 4, 8, 16))}
        return d

    def xscale(self):
        """Section 3.4 activation factors [K] in clustered order (1.0 if the
        layer is not scaled)."""
        out = np.empty(self.info()["K"], np.float32)
        _check(_lib.polyq_layer_xscale(self._h, out.ctypes.data))
        return out

    def export(self, meta_stride=None) -> dict:
        """Host copies; meta rows have ``meta_stride`` entries (default: the
        compact n_groups; pass info()['meta_stride'] for the device layout)."""
        inf = self.info()
        N, K, S, G = inf["N"], inf["K"], inf["row_stride"], inf["n_groups"]
        ms = G if meta_stride is None else int(meta_stride)
        packed = np.empty((N, S), np.uint8)
        meta = np.empty((N, ms), np.uint32)
        perm = np.empty(K, np.int32)
        bits = np.empty(K, np.uint8)
        out_perm = np.empty(N, np.int32)
        _check(_lib.polyq_layer_export(self._h, packed.ctypes.data, meta.ctypes.data, ms,
                                       perm.ctypes.data, bits.ctypes.data, out_perm.ctypes.data))
        return dict(info=inf, packed=packed, meta=meta, perm=perm, bits=bits, out_perm=out_perm)

    def permute_rows(self, row_perm):
        """Reorder the output rows (Section 4.3 merge): row i becomes old row row_perm[i]."""
        rp = np.ascontiguousarray(row_perm, dtype=np.int32)
        _check(_lib.polyq_layer_permute_rows(self._h, rp.ctypes.data))


class DeviceLayer:
    """Device copy of a packed layer (torch tensors) and its descriptor."""

    def __init__(self, host: HostLayer, device="cuda", gather=None, identity_gather=False):
        import torch
        ex = host.export(meta_stride=host.info()["meta_stride"])
        self.info = ex["info"]
        self.perm = ex["perm"]
        self.out_perm = ex["out_perm"]
        self.packed = torch.from_numpy(ex["packed"]).to(device)
        self.meta = torch.from_numpy(ex["meta"].view(np.int32)).to(device)
        if identity_gather:
            self.gather = None
        else:
            g = ex["perm"] if gather is None else np.ascontiguousarray(gather, np.int32)
            self.gather = torch.from_numpy(np.ascontiguousarray(g, np.int32)).to(device)
        self.desc = DevLayer()
        _check(_lib.polyq_dev_layer_fill(
            host._h, self.packed.data_ptr(), self.meta.data_ptr() if self.meta.numel() else None,
            self.gather.data_ptr() if self.gather is not None else None, C.byref(self.desc)))
        self.xscale = None
        if self.info["has_xscale"]:
            self.xscale = torch.from_numpy(host.xscale()).to(device)
            self.desc.xscale = self.xscale.data_ptr()
        self.N = self.info["N"]
        self.K = self.info["K"]

    def packed_bytes(self):
        """Device bytes of the packed codes and their scale/zero metadata."""
        return self.info["packed_bytes"] + self.info["meta_bytes"]

    def clone(self):
        """A second device copy of the same packed layer (distinct memory)."""
        c = object.__new__(DeviceLayer)
        c.info, c.perm, c.out_perm, c.N, c.K = self.info, self.perm, self.out_perm, self.N, self.K
        c.xscale = self.xscale
        c.packed = self.packed.clone()
        c.meta = self.meta.clone()
        c.gather = self.gather
        c.desc = DevLayer()
        C.pointer(c.desc)[0] = self.desc
        c.desc.packed = c.packed.data_ptr()
        c.desc.meta = c.meta.data_ptr() if c.meta.numel() else None
        return c


def _require(t, name, dtype, shape, device):
    """ValueError unless `t` is a contiguous tensor of `dtype` and `shape` on
    `device`: the library reads and writes through raw pointers, so a wrong
    buffer would otherwise reach the GPU."""
    import torch
    if (not isinstance(t, torch.Tensor) or t.dtype != dtype or tuple(t.shape) != tuple(shape)
            or t.device != device or not t.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous {dtype} tensor {list(shape)} on {device}")


def _cuda_input(x, name, dtype, K):
    """Checks a [rows][K] CUDA input of `dtype` and returns its device, which
    must be the current device: the stream and the library's per-device state
    are looked up for the current device."""
    import torch
    if (not isinstance(x, torch.Tensor) or x.dtype != dtype or not x.is_cuda or x.dim() != 2
            or x.shape[1] != K):
        raise ValueError(f"{name} must be a CUDA {dtype} tensor [rows][{K}]")
    if x.device.index != torch.cuda.current_device():
        raise ValueError(f"{name} is on {x.device}, not on the current device "
                         f"cuda:{torch.cuda.current_device()}")
    return x.device


def _stream_ptr(stream):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return C.c_void_p(s.cuda_stream)


def gemv_workspace_bytes(layer: DeviceLayer, batch: int) -> int:
    """Workspace bytes one GEMV call on `layer` at `batch` needs."""
    n = C.c_size_t()
    _check(_lib.polyq_gemv_workspace_bytes(C.byref(layer.desc), int(batch), C.byref(n)))
    return n.value


def linear_gemv(layer: DeviceLayer, x, y=None, residual=None, workspace=None, stream=None):
    """y[b][n] = residual[b][n] + sum_p x[b][gather[p]] W'[n][p] (device tensors)."""
    import torch
    dev = _cuda_input(x, "x", torch.bfloat16, layer.K)
    x = x.contiguous()
    batch = x.shape[0]
    if y is None:
        y = torch.empty((batch, layer.N), dtype=torch.float32, device=dev)
    _require(y, "y", torch.float32, (batch, layer.N), dev)
    if residual is not None:
        _require(residual, "residual", torch.float32, (batch, layer.N), dev)
    ws_need = gemv_workspace_bytes(layer, batch)
    if workspace is None and ws_need:
        # the status word must start at zero; every call rewrites the records
        workspace = torch.zeros(ws_need, dtype=torch.uint8, device=dev)
    if workspace is not None:
        _require(workspace, "workspace", torch.uint8, (workspace.numel(),), dev)
    ws_ptr = workspace.data_ptr() if workspace is not None else None
    ws_len = workspace.numel() if workspace is not None else 0
    _check(_lib.polyq_linear_gemv(C.byref(layer.desc), x.data_ptr(), batch, y.data_ptr(),
                                  residual.data_ptr() if residual is not None else None,
                                  ws_ptr, ws_len, _stream_ptr(stream)))
    return y


def linear_gemv_noalloc(layer: DeviceLayer, x, y, residual=None, stream=None):
    """linear_gemv on the library's fixed scratch array, for callers that cannot
    allocate device memory (a plugin whose host program owns the device through
    its own pool, or a loop that cannot take cudaMalloc's device-wide sync).

    `y` must be passed: nothing is allocated here.  Calls that may overlap on
    the GPU share the scratch and race; the first call on a device looks up the
    scratch address and should come before any stream capture there.  Read
    noalloc_status() after a call to learn whether a bounded device wait gave
    up.
    """
    import torch
    dev = _cuda_input(x, "x", torch.bfloat16, layer.K)
    if not x.is_contiguous():
        raise ValueError("x must be contiguous (no copy is made here)")
    batch = x.shape[0]
    _require(y, "y", torch.float32, (batch, layer.N), dev)
    if residual is not None:
        _require(residual, "residual", torch.float32, (batch, layer.N), dev)
    _check(_lib.polyq_linear_gemv_noalloc(C.byref(layer.desc), x.data_ptr(), batch, y.data_ptr(),
                                          residual.data_ptr() if residual is not None else None,
                                          _stream_ptr(stream)))
    return y


def noalloc_status(stream=None):
    """Status word of the current device's no-allocation scratch after the
    queued work: 0 when the last linear_gemv_noalloc call's waits all
    completed; raises PolyqError(POLYQ_ETIMEOUT) when one gave up."""
    v = C.c_int()
    _check(_lib.polyq_noalloc_status(C.byref(v), _stream_ptr(stream)))
    return v.value


def _layer_array(layers):
    arr = (C.POINTER(DevLayer) * len(layers))()
    for i, l in enumerate(layers):
        arr[i] = C.pointer(l.desc)
    return arr


def gemv_group_workspace_bytes(layers, batch: int) -> int:
    """Workspace bytes one grouped GEMV call on `layers` at `batch` needs."""
    n = C.c_size_t()
    _check(_lib.polyq_gemv_group_workspace_bytes(_layer_array(layers), len(layers), int(batch),
                                                 C.byref(n)))
    return n.value


def _check_outputs(layers, batch, ys, residuals, dev):
    import torch
    if len(ys) != len(layers) or (residuals is not None and len(residuals) != len(layers)):
        raise ValueError("one y (and one residual, or None) per layer")
    for i, l in enumerate(layers):
        _require(ys[i], f"ys[{i}]", torch.float32, (batch, l.N), dev)
        if residuals is not None and residuals[i] is not None:
            _require(residuals[i], f"residuals[{i}]", torch.float32, (batch, l.N), dev)


def linear_gemv_group(layers, xs, ys=None, residuals=None, workspace=None, stream=None):
    """Independent GEMVs in one launch: ys[i] = residuals[i] + xs[i] W_i'^T."""
    import torch
    n = len(layers)
    if len(xs) != n:
        raise ValueError("one x per layer")
    batch = xs[0].shape[0]
    dev = None
    for l, x in zip(layers, xs):
        d = _cuda_input(x, "each x", torch.bfloat16, l.K)
        if x.shape[0] != batch or (dev is not None and d != dev):
            raise ValueError("every x must have the same batch and device")
        dev = d
    xs = [x.contiguous() for x in xs]
    if ys is None:
        ys = [torch.empty((batch, l.N), dtype=torch.float32, device=dev) for l in layers]
    _check_outputs(layers, batch, ys, residuals, dev)
    need = gemv_group_workspace_bytes(layers, batch)
    if workspace is None:
        workspace = torch.zeros(need, dtype=torch.uint8, device=dev)
    _require(workspace, "workspace", torch.uint8, (workspace.numel(),), dev)
    xa = (C.c_void_p * n)(*[x.data_ptr() for x in xs])
    ya = (C.c_void_p * n)(*[y.data_ptr() for y in ys])
    ra = None
    if residuals is not None:
        ra = (C.c_void_p * n)(*[r.data_ptr() if r is not None else None for r in residuals])
    _check(_lib.polyq_linear_gemv_group(_layer_array(layers), n, xa, batch, ya, ra,
                                        workspace.data_ptr(), workspace.numel(),
                                        _stream_ptr(stream)))
    return ys


def linear_gemv_input(layers, kind, a, b=None, eps=1e-6, ys=None, residuals=None, x_out=None,
                      workspace=None, stream=None):
    """GEMVs of `layers` on one shared input with its transform fused into the
    pre-pass (X_BF16, X_F32, X_RMSNORM or X_SILU_MUL, see polyq.h)."""
    import torch
    n = len(layers)
    K = layers[0].K
    want = torch.bfloat16 if kind == X_BF16 else torch.float32
    dev = _cuda_input(a, "a", want, K)
    if not a.is_contiguous():
        raise ValueError("a must be contiguous")
    batch = a.shape[0]
    if (kind == X_SILU_MUL) != (b is not None):
        raise ValueError("b is the second input of X_SILU_MUL only")
    if b is not None:
        _require(b, "b", torch.float32, tuple(a.shape), dev)
    if x_out is not None:
        _require(x_out, "x_out", torch.bfloat16, tuple(a.shape), dev)
    if ys is None:
        ys = [torch.empty((batch, l.N), dtype=torch.float32, device=dev) for l in layers]
    _check_outputs(layers, batch, ys, residuals, dev)
    need = gemv_group_workspace_bytes(layers, batch)
    if workspace is None:
        workspace = torch.zeros(need, dtype=torch.uint8, device=dev)
    _require(workspace, "workspace", torch.uint8, (workspace.numel(),), dev)
    inp = GemvInput(kind, eps, a.data_ptr(), b.data_ptr() if b is not None else None,
                    x_out.data_ptr() if x_out is not None else None)
    ya = (C.c_void_p * n)(*[y.data_ptr() for y in ys])
    ra = None
    if residuals is not None:
        ra = (C.c_void_p * n)(*[r.data_ptr() if r is not None else None for r in residuals])
    _check(_lib.polyq_linear_gemv_input(_layer_array(layers), n, C.byref(inp), batch, ya, ra,
                                        workspace.data_ptr(), workspace.numel(),
                                        _stream_ptr(stream)))
    return ys


def gemm_workspace_bytes(layer: DeviceLayer, M: int) -> int:
    """Workspace bytes one GEMM call on `layer` with M tokens needs."""
    n = C.c_size_t()
    _check(_lib.polyq_gemm_workspace_bytes(C.byref(layer.desc), int(M), C.byref(n)))
    return n.value


def linear_gemm(layer: DeviceLayer, X, Y=None, workspace=None, stream=None):
    """Y[m][n] = sum_p X[m][gather[p]] W'[n][p] (device tensors)."""
    import torch
    dev = _cuda_input(X, "X", torch.bfloat16, layer.K)
    X = X.contiguous()
    M = X.shape[0]
    if Y is None:
        Y = torch.empty((M, layer.N), dtype=torch.float32, device=dev)
    _require(Y, "Y", torch.float32, (M, layer.N), dev)
    ws_need = gemm_workspace_bytes(layer, M)
    if workspace is None and ws_need:
        workspace = torch.empty(ws_need, dtype=torch.uint8, device=dev)
    if workspace is not None:
        _require(workspace, "workspace", torch.uint8, (workspace.numel(),), dev)
    ws_ptr = workspace.data_ptr() if workspace is not None else None
    ws_len = workspace.numel() if workspace is not None else 0
    _check(_lib.polyq_linear_gemm(C.byref(layer.desc), X.data_ptr(), M, Y.data_ptr(),
                                  ws_ptr, ws_len, _stream_ptr(stream)))
    return Y


def unpack_codes(layer: DeviceLayer, stream=None):
    """Device-unpacked integer codes [N][K] (clustered order) as numpy uint16."""
    import torch
    out = torch.empty((layer.N, layer.K), dtype=torch.int16, device=layer.packed.device)
    _check(_lib.polyq_unpack_codes(C.byref(layer.desc), out.data_ptr(), _stream_ptr(stream)))
    torch.cuda.synchronize()
    return out.cpu().numpy().view(np.uint16)


def gemv_launches_per_call(layer: DeviceLayer, batch: int) -> int:
    """Kernels one polyq_linear_gemv (or _group) call enqueues: the activation
    record pre-pass and the streaming kernel."""
    return 2


def decoder_plan_graph(n_layers, hidden, ffn, perm_of, kv=None, qdim=None, free_source=False,
                       head=None):
    """Planner input for a decoder stack's decode step: per layer RMSNorm ->
    q, k, v -> attention -> o -> residual add -> RMSNorm -> gate, up ->
    SiLU * up -> down -> residual add; by default the stream enters in
    natural order and leaves through a natural-order boundary.
    ``free_source``: it enters from an embedding whose columns may be
    permuted (any order at no cost).  ``head = (perm id, vocab)``: it ends in
    a final RMSNorm and an output-head linear whose logits leave through a
    boundary.  ``perm_of(layer, name)`` returns the permutation id of each
    linear.  Returns (nodes, edge widths, per-layer edge ids by name)."""
    qdim = hidden if qdim is None else qdim
    kv = qdim if kv is None else kv
    nodes, dims, names = [], [], []

    def edge(w):
        dims.append(w)
        return len(dims) - 1

    s = edge(hidden)
    nodes.append((NODE_SOURCE_FREE if free_source else NODE_SOURCE_FIXED, [], s, -1))
    for l in range(n_layers):
        e = {"s_in": s, "h": edge(hidden)}
        nodes.append((NODE_ELEMENTWISE, [s], e["h"], -1))
        for nm, w in (("q", qdim), ("k", kv), ("v", kv)):
            e[nm] = edge(w)
            nodes.append((NODE_LINEAR, [e["h"]], e[nm], perm_of(l, nm)))
        e["att"] = edge(qdim)
        nodes.append((NODE_ATTENTION, [e["q"], e["k"], e["v"]], e["att"], -1))
        e["o"] = edge(hidden)
        nodes.append((NODE_LINEAR, [e["att"]], e["o"], perm_of(l, "o")))
        e["s1"] = edge(hidden)
        nodes.append((NODE_ELEMENTWISE, [s, e["o"]], e["s1"], -1))
        e["h2"] = edge(hidden)
        nodes.append((NODE_ELEMENTWISE, [e["s1"]], e["h2"], -1))
        for nm in ("gate", "up"):
            e[nm] = edge(ffn)
            nodes.append((NODE_LINEAR, [e["h2"]], e[nm], perm_of(l, nm)))
        e["m"] = edge(ffn)
        nodes.append((NODE_ELEMENTWISE, [e["gate"], e["up"]], e["m"], -1))
        e["down"] = edge(hidden)
        nodes.append((NODE_LINEAR, [e["m"]], e["down"], perm_of(l, "down")))
        e["s2"] = edge(hidden)
        nodes.append((NODE_ELEMENTWISE, [e["s1"], e["down"]], e["s2"], -1))
        names.append(e)
        s = e["s2"]
    if head is None:
        nodes.append((NODE_BOUNDARY, [s], -1, -1))
    else:
        hf = edge(hidden)
        nodes.append((NODE_ELEMENTWISE, [s], hf, -1))  # final RMSNorm
        logits = edge(head[1])
        nodes.append((NODE_LINEAR, [hf], logits, head[0]))
        nodes.append((NODE_BOUNDARY, [logits], -1, -1))
    return nodes, dims, names


class GemvChain:
    """A chain of dependent GEMV phases run in one persistent launch
    (polyq_linear_gemv_chain).  Each phase is a dict with ``layers`` (one to
    eight DeviceLayer reading one input), ``kind`` (X_BF16, X_F32, X_RMSNORM,
    X_SILU_MUL), ``a`` (and ``b`` for X_SILU_MUL) CUDA tensors [batch][K],
    ``ys`` fp32 CUDA tensors [batch][N], optional ``residuals``, ``eps``,
    ``x_out`` and, for X_BF16, per-layer inputs ``xs``.  The tensors must
    stay alive and in place while the chain is used."""

    def __init__(self, phases, batch, stream=None):
        import torch
        self._keep = []
        arr = (GemvPhase * len(phases))()
        for i, ph in enumerate(phases):
            layers = ph["layers"]
            arr[i].n_layers = len(layers)
            for j, L in enumerate(layers):
                arr[i].layers[j] = C.pointer(L.desc)
                self._keep.append(L)
            kind = ph.get("kind", X_BF16)
            a, b, xo = ph.get("a"), ph.get("b"), ph.get("x_out")
            arr[i].in_ = GemvInput(kind, float(ph.get("eps", 1e-6)),
                                   a.data_ptr() if a is not None else None,
                                   b.data_ptr() if b is not None else None,
                                   xo.data_ptr() if xo is not None else None)
            for j, x in enumerate(ph.get("xs") or []):
                arr[i].xs[j] = x.data_ptr() if x is not None else None
            for j, y in enumerate(ph["ys"]):
                arr[i].ys[j] = y.data_ptr()
            for j, r in enumerate(ph.get("residuals") or []):
                arr[i].residuals[j] = r.data_ptr() if r is not None else None
            self._keep.append(ph)
        h = C.c_void_p()
        _check(_lib.polyq_gemv_chain_create(arr, len(phases), int(batch), C.byref(h)))
        self._h = h
        nbytes = C.c_size_t()
        _check(_lib.polyq_gemv_chain_plan_bytes(self._h, C.byref(nbytes)))
        self.plan = torch.empty(max(1, nbytes.value), dtype=torch.uint8, device="cuda")
        _check(_lib.polyq_gemv_chain_upload(self._h, self.plan.data_ptr(), self.plan.numel(),
                                            _stream_ptr(stream)))
        wsb = C.c_size_t()
        _check(_lib.polyq_gemv_chain_workspace_bytes(self._h, C.byref(wsb)))
        self.workspace = torch.zeros(wsb.value, dtype=torch.uint8, device="cuda")
        self.n_phases = len(phases)

    def run(self, stream=None, workspace=None):
        """Launch every phase of the chain once on `stream` (one cooperative launch)."""
        ws = self.workspace if workspace is None else workspace
        _check(_lib.polyq_linear_gemv_chain(self._h, ws.data_ptr(), ws.numel(),
                                            _stream_ptr(stream)))

    def __del__(self):
        if getattr(self, "_h", None) and self._h.value:
            _lib.polyq_gemv_chain_free(self._h)
            self._h = C.c_void_p()


def workspace_status(workspace, stream=None):
    """Status word of a workspace after the queued work (0: no device wait
    gave up); raises PolyqError(POLYQ_ETIMEOUT) when one did."""
    v = C.c_int()
    _check(_lib.polyq_workspace_status(workspace.data_ptr(), C.byref(v), _stream_ptr(stream)))
    return v.value
