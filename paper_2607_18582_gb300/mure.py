"""Thin ctypes binding of libmure.so (include/mure.h).

Argument marshalling only: every step of the method runs in the library's CUDA
kernels.  Functions carry the C names.  PyTorch supplies device memory (its caching
allocator is handed to the library) and the CUDA stream.  There is no fallback: if
the library has not been built, every call raises.
"""
from __future__ import annotations

import ctypes as C
import os
import sys

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libmure.so")

STATUS = {0: "MURE_OK", 1: "MURE_ERR_INVALID_ARG", 2: "MURE_ERR_UNSUPPORTED", 3: "MURE_ERR_OOM",
          4: "MURE_ERR_CUDA", 5: "MURE_ERR_TIMEOUT"}
KINDS = {"conv": 0, "dense": 1, "maxpool": 2, "flatten": 3, "add": 4, "gap": 5, "shortcut": 6, "dwconv": 7,
         "embed": 8, "lstm": 9}
ACTS = {"none": 0, "relu": 1, "relu6": 2}
PRECISIONS = {"fp32": 0, "tf32x3": 1, "bf16": 2, "tf32": 3}

# the exported entry points of include/mure.h
EXPORTS = ("mure_create", "mure_destroy", "mure_last_error", "mure_model_load", "mure_model_free",
           "mure_model_n_layers", "mure_model_layer_kernel", "mure_kernel_launches", "mure_build_prefix_cache", "mure_cache_free", "mure_cache_outputs",
           "mure_eval_mutants", "mure_eval_vanilla", "mure_expand_patches", "mure_expand_patches_noalloc",
           "mure_check_descriptors", "mure_set_wait_limit")


class MureError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class _Node(C.Structure):
    _fields_ = [("kind", C.c_int32), ("act", C.c_int32), ("in0", C.c_int32), ("in1", C.c_int32),
                ("kh", C.c_int32), ("kw", C.c_int32), ("stride", C.c_int32), ("pad", C.c_int32),
                ("cin", C.c_int32), ("cout", C.c_int32), ("W", C.c_void_p), ("b", C.c_void_p)]


class _ModelDesc(C.Structure):
    _fields_ = [("in_h", C.c_int32), ("in_w", C.c_int32), ("in_c", C.c_int32), ("n_classes", C.c_int32),
                ("n_nodes", C.c_int32), ("precision", C.c_int32), ("nodes", C.POINTER(_Node))]


MUTANT_DTYPE = np.dtype([("layer", "<i4"), ("op", "<i4"), ("n_neurons", "<i4"), ("tagged", "<i4"),
                         ("neuron_off", "<i8"), ("param", "<f4"), ("reserved2", "<f4"), ("seed", "<u8")])

_ALLOC_FN = C.CFUNCTYPE(C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p)
_FREE_FN = C.CFUNCTYPE(None, C.c_void_p, C.c_void_p, C.c_void_p)


class _Allocator(C.Structure):
    _fields_ = [("alloc", _ALLOC_FN), ("free", _FREE_FN), ("user", C.c_void_p)]


class _Opts(C.Structure):
    _fields_ = [("outputs_on_device", C.c_int32), ("kernel_timing", C.c_int32), ("workspace_bytes", C.c_int64),
                ("logits_out", C.c_void_p), ("skip_unchanged", C.c_int32), ("reserved", C.c_int32)]


class _Stats(C.Structure):
    _fields_ = [("ms_total", C.c_double), ("ms_expand", C.c_double), ("ms_suffix", C.c_double),
                ("ms_score", C.c_double), ("n_rows", C.c_int64), ("n_near_ties", C.c_int64),
                ("n_groups", C.c_int64), ("n_batches", C.c_int64), ("kernel_launches", C.c_int64),
                ("flops", C.c_int64), ("ms_layer", C.c_double * 64), ("flops_layer", C.c_int64 * 64),
                ("launches_layer", C.c_int64 * 64), ("ms_delta", C.c_double), ("ms_delta_values", C.c_double),
                ("ms_epilogue", C.c_double), ("bytes_gather", C.c_int64), ("launches_delta", C.c_int64),
                ("bytes_rows", C.c_int64), ("n_rows_unchanged", C.c_int64), ("launches_delta_values", C.c_int64),
                ("bytes_delta_values", C.c_int64)]

    def as_dict(self):
        out = {}
        for k, _ in self._fields_:
            v = getattr(self, k)
            out[k] = list(v) if hasattr(v, "__len__") else v
        return out


_lib = None
# Allocator thunks stay alive for the life of the process: a context's C object may
# still call them while Python tears objects down in arbitrary (cyclic-GC) order.
_ALLOCATOR_KEEPALIVE = []


def _finalizing():
    return sys is None or sys.is_finalizing()


def lib():
    """The loaded library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libmure.so is not built ({LIB_PATH}); run __graft_entry__.build() "
                               "or python paper_2607_18582_gb300/build.py")
        L = C.CDLL(LIB_PATH)
        vp, i64, i32 = C.c_void_p, C.c_int64, C.c_int32
        L.mure_create.argtypes = [C.c_int, vp, C.POINTER(_Allocator), C.POINTER(vp)]
        L.mure_destroy.argtypes = [vp]
        L.mure_destroy.restype = None
        L.mure_last_error.argtypes = [vp]
        L.mure_last_error.restype = C.c_char_p
        L.mure_model_load.argtypes = [vp, C.POINTER(_ModelDesc), C.POINTER(vp)]
        L.mure_model_free.argtypes = [vp]
        L.mure_model_free.restype = None
        L.mure_model_n_layers.argtypes = [vp]
        L.mure_model_n_layers.restype = i32
        L.mure_model_layer_kernel.argtypes = [vp, i32, C.POINTER(i32), C.POINTER(i64)]
        L.mure_kernel_launches.argtypes = [vp]
        L.mure_kernel_launches.restype = i64
        L.mure_build_prefix_cache.argtypes = [vp, vp, i64, vp, C.c_int, C.POINTER(vp)]
        L.mure_cache_free.argtypes = [vp]
        L.mure_cache_free.restype = None
        L.mure_cache_outputs.argtypes = [vp, vp, vp]
        L.mure_eval_mutants.argtypes = [vp, vp, i64, vp, i64, C.POINTER(_Opts), vp, C.POINTER(C.c_double),
                                        C.POINTER(C.c_double), C.POINTER(_Stats)]
        L.mure_eval_vanilla.argtypes = [vp, vp, i64, vp, C.c_int, vp, i64, vp, i64, C.POINTER(_Opts), vp,
                                        C.POINTER(C.c_double), C.POINTER(C.c_double), C.POINTER(_Stats)]
        L.mure_expand_patches.argtypes = [vp, vp, i64, vp, i64, vp, i64, vp]
        L.mure_expand_patches_noalloc.argtypes = [vp, vp, i64, vp, i64, vp, i64, vp]
        L.mure_check_descriptors.argtypes = [C.POINTER(_ModelDesc), vp, i64, vp, i64, C.c_char_p, C.c_size_t]
        L.mure_set_wait_limit.argtypes = [vp, i64]
        for name in EXPORTS:
            if name not in ("mure_destroy", "mure_model_free", "mure_cache_free", "mure_last_error",
                            "mure_model_n_layers", "mure_kernel_launches"):
                getattr(L, name).restype = C.c_int
        _lib = L
    return _lib


def _ptr(a):
    """Address of a numpy array or a torch tensor (None -> NULL)."""
    if a is None:
        return None
    if hasattr(a, "data_ptr"):
        return a.data_ptr()
    return a.ctypes.data


def _is_device(a):
    return a is not None and hasattr(a, "is_cuda") and a.is_cuda


class Context:
    """Owns a library context.  Models and caches made from it count as children; the
    C context is destroyed only once none is alive (and never during interpreter
    shutdown, when the process frees everything anyway)."""

    def __init__(self, handle, keep):
        self.h = handle
        self._keep = keep
        self._children = 0
        self._released = False

    def check(self, status):
        if status != 0:
            msg = lib().mure_last_error(self.h)
            raise MureError(status, msg.decode() if msg else "")

    def _child_gone(self):
        self._children -= 1
        if self._released and self._children == 0:
            self._destroy()

    def _destroy(self):
        if self.h and not _finalizing():
            lib().mure_destroy(self.h)
        self.h = None

    def __del__(self):
        self._released = True
        if getattr(self, "h", None) and self._children == 0:
            self._destroy()


def mure_create(device: int = 0, stream=None, torch_allocator: bool = True) -> Context:
    """A library context on `device` queueing on `stream` (default: torch's current
    stream), allocating through torch's caching allocator."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(device)
    handle_stream = stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream or 0)
    keep = []
    alloc_p = None
    if torch_allocator:
        def _alloc(nbytes, strm, user):
            try:
                return torch.cuda.caching_allocator_alloc(int(nbytes), device, int(strm or 0))
            except Exception:  # noqa: BLE001 - reported to the library as a NULL allocation
                return None

        def _free(ptr, strm, user):
            torch.cuda.caching_allocator_delete(ptr)

        def _free_guarded(ptr, strm, user):
            if not _finalizing():
                _free(ptr, strm, user)

        a = _Allocator(_ALLOC_FN(_alloc), _FREE_FN(_free_guarded), None)
        keep += [a, a.alloc, a.free]
        _ALLOCATOR_KEEPALIVE.append(keep)
        alloc_p = C.byref(a)
    out = C.c_void_p()
    st = lib().mure_create(device, handle_stream, alloc_p, C.byref(out))
    if st != 0:
        raise MureError(st, "mure_create failed")
    return Context(out.value, keep)


class Model:
    def __init__(self, ctx, handle, src):
        self.ctx, self.h, self.src = ctx, handle, src
        ctx._children += 1
        self._children = 0
        self._released = False

    @property
    def n_layers(self):
        return lib().mure_model_n_layers(self.h)

    KERNELS = {0: "simt_gemm", 1: "simt_small", 2: "tc_gemm", 3: "tc_window", 4: "output", 5: "tc_conv"}

    def layer_kernel(self, layer):
        """(kernel name, executed multiply-accumulates per batch row) of a layer."""
        k, macs = C.c_int32(), C.c_int64()
        self.ctx.check(lib().mure_model_layer_kernel(self.h, int(layer), C.byref(k), C.byref(macs)))
        return self.KERNELS.get(k.value, str(k.value)), macs.value

    def _child_gone(self):
        self._children -= 1
        if self._released and self._children == 0:
            self._destroy()

    def _destroy(self):
        if self.h:
            if not _finalizing():
                lib().mure_model_free(self.h)
            self.h = None
            self.ctx._child_gone()

    def __del__(self):
        self._released = True
        if getattr(self, "h", None) and self._children == 0:
            self._destroy()


def _model_desc(model, precision):
    """The C description of a network (workloads.Model fields) and the arrays it points to."""
    nodes = (_Node * len(model.nodes))()
    keep = []
    for v, n in enumerate(model.nodes):
        W = None if n.W is None else np.ascontiguousarray(n.W, np.float32)
        b = None if n.b is None else np.ascontiguousarray(n.b, np.float32)
        keep += [W, b]
        ins = list(n.inputs) + [-1] * (2 - len(n.inputs))
        nodes[v] = _Node(KINDS[n.kind], ACTS[n.act], ins[0], ins[1], n.kh, n.kw, n.stride, n.pad, n.cin, n.cout,
                         _ptr(W), _ptr(b))
    h, w, c = model.in_shape
    desc = _ModelDesc(h, w, c, model.n_classes, len(model.nodes), PRECISIONS[precision], nodes)
    return desc, (keep, nodes)


def mure_model_load(ctx: Context, model, precision: str = "fp32") -> Model:
    """Copy a network description (workloads.Model fields) to the device."""
    desc, keep = _model_desc(model, precision)
    out = C.c_void_p()
    ctx.check(lib().mure_model_load(ctx.h, C.byref(desc), C.byref(out)))
    return Model(ctx, out.value, model)


class Cache:
    def __init__(self, model, handle, n_inputs):
        self.model, self.h, self.n_inputs = model, handle, n_inputs
        model._children += 1

    def free(self):
        if getattr(self, "h", None):
            if not _finalizing():
                lib().mure_cache_free(self.h)
            self.h = None
            self.model._child_gone()

    def __del__(self):
        self.free()


def _as_input(X, labels):
    on_dev = _is_device(X)
    if not on_dev:
        X = np.ascontiguousarray(X, np.float32)
        if labels is not None:
            labels = np.ascontiguousarray(labels, np.int32)
    else:
        X = X.contiguous()
        if labels is not None:
            import torch
            labels = labels.to(device=X.device, dtype=torch.int32).contiguous()
    return X, labels, int(on_dev)


def mure_build_prefix_cache(model: Model, X, labels=None) -> Cache:
    """Prefix-activation cache of X (numpy host array or CUDA tensor, NHWC fp32)."""
    X, labels, on_dev = _as_input(X, labels)
    n = int(X.shape[0])
    out = C.c_void_p()
    model.ctx.check(lib().mure_build_prefix_cache(model.h, _ptr(X) if n else None, n, _ptr(labels), on_dev,
                                                  C.byref(out)))
    return Cache(model, out.value, n)


def mure_cache_outputs(cache: Cache):
    """(original logits [n][C], original predictions [n]) held by the cache."""
    C_ = cache.model.src.n_classes
    lg = np.zeros((cache.n_inputs, C_), np.float32)
    pr = np.zeros(cache.n_inputs, np.int32)
    cache.model.ctx.check(lib().mure_cache_outputs(cache.h, _ptr(lg), _ptr(pr)))
    return lg, pr


def table_array(table):
    """A workloads.MutantTable as the C descriptor array and the neuron pool."""
    n = len(table)
    arr = np.zeros(max(n, 1), MUTANT_DTYPE)
    arr["layer"][:n] = table.layer
    arr["op"][:n] = table.op
    arr["n_neurons"][:n] = table.n_neurons
    arr["neuron_off"][:n] = table.neuron_off
    arr["param"][:n] = table.param
    arr["seed"][:n] = table.seed
    if getattr(table, "tagged", None) is not None:
        arr["tagged"][:n] = table.tagged
    pool = np.ascontiguousarray(table.pool, np.int32)
    if pool.size == 0:
        pool = np.zeros(1, np.int32)
    return arr, pool, int(table.pool.size)


def _eval_common(n_mut, n_in, n_classes, logits, outputs_on_device, workspace_bytes, kill_out, kernel_timing=False,
                 skip_unchanged=False):
    W64 = (n_in + 63) // 64
    if outputs_on_device:
        import torch
        kill = kill_out if kill_out is not None else torch.empty((max(n_mut, 1), max(W64, 1)), dtype=torch.int64,
                                                                 device="cuda")
        lg = torch.empty((n_mut, n_in, n_classes), dtype=torch.float32, device="cuda") if logits else None
    else:
        kill = kill_out if kill_out is not None else np.zeros((max(n_mut, 1), max(W64, 1)), np.uint64)
        lg = np.zeros((n_mut, n_in, n_classes), np.float32) if logits else None
    opts = _Opts(int(bool(outputs_on_device)), int(bool(kernel_timing)), int(workspace_bytes), _ptr(lg),
                 int(bool(skip_unchanged)), 0)
    return kill, lg, opts, W64


def _eval_result(kill, lg, sa, sb, st, n_mut, W64, outputs_on_device):
    if outputs_on_device:
        kill = kill[:n_mut, :W64]
    else:
        kill = kill[:n_mut, :W64]
    return {"kill_bits": kill, "scoreA": sa.value, "scoreB": sb.value, "stats": st.as_dict(), "logits": lg}


def mure_eval_mutants(cache: Cache, table, logits: bool = False, outputs_on_device: bool = False,
                      workspace_bytes: int = 0, kill_out=None, kernel_timing: bool = False, arrays=None,
                      skip_unchanged: bool = False):
    """Memoized mutation testing of `table` on the cached inputs (skip_unchanged: the
    exact unchanged-row elimination)."""
    arr, pool, plen = arrays if arrays is not None else table_array(table)
    n = len(table)
    kill, lg, opts, W64 = _eval_common(n, cache.n_inputs, cache.model.src.n_classes, logits, outputs_on_device,
                                       workspace_bytes, kill_out, kernel_timing, skip_unchanged)
    sa, sb, st = C.c_double(), C.c_double(), _Stats()
    cache.model.ctx.check(lib().mure_eval_mutants(cache.h, _ptr(arr), n, _ptr(pool), plen, C.byref(opts), _ptr(kill),
                                                  C.byref(sa), C.byref(sb), C.byref(st)))
    return _eval_result(kill, lg, sa, sb, st, n, W64, outputs_on_device)


def mure_eval_vanilla(model: Model, X, table, labels=None, logits: bool = False, outputs_on_device: bool = False,
                      workspace_bytes: int = 0, kill_out=None, kernel_timing: bool = False):
    """Vanilla mutation testing: every mutant end to end from X."""
    X, labels, on_dev = _as_input(X, labels)
    arr, pool, plen = table_array(table)
    n = len(table)
    n_in = int(X.shape[0])
    kill, lg, opts, W64 = _eval_common(n, n_in, model.src.n_classes, logits, outputs_on_device, workspace_bytes,
                                       kill_out, kernel_timing)
    sa, sb, st = C.c_double(), C.c_double(), _Stats()
    model.ctx.check(lib().mure_eval_vanilla(model.h, _ptr(X) if n_in else None, n_in, _ptr(labels), on_dev, _ptr(arr),
                                            n, _ptr(pool), plen, C.byref(opts), _ptr(kill), C.byref(sa), C.byref(sb),
                                            C.byref(st)))
    return _eval_result(kill, lg, sa, sb, st, n, W64, outputs_on_device)


def mure_kernel_launches(ctx: Context) -> int:
    """Kernels the context has launched since it was created."""
    return int(lib().mure_kernel_launches(ctx.h))


def mure_set_wait_limit(ctx: Context, cycles: int) -> None:
    """Limit of the tensor-core kernels' device-side waits in SM cycles (0: default)."""
    ctx.check(lib().mure_set_wait_limit(ctx.h, int(cycles)))


def mure_expand_patches(model: Model, table):
    """GF noise / WS-permuted weights of every GF or WS mutant: (values, offsets)."""
    arr, pool, plen = table_array(table)
    n = len(table)
    need = 0
    for i in range(n):
        if int(table.op[i]) in (0, 4):
            layer = model.src.nodes[model.src.layers()[int(table.layer[i])]]
            fan = layer.kh * layer.kw * layer.cin if layer.kind == "conv" else layer.cin
            need += int(table.n_neurons[i]) * fan
    out = np.zeros(max(need, 1), np.float32)
    offs = np.zeros(max(n, 1), np.int64)
    model.ctx.check(lib().mure_expand_patches(model.h, _ptr(arr), n, _ptr(pool), plen, _ptr(out), need, _ptr(offs)))
    return out[:need], offs[:n]


def mure_expand_patches_noalloc(model: Model, table, out_dev):
    """mure_expand_patches into a caller-provided CUDA float32 tensor, with no device
    allocation by the library; returns the offsets (host)."""
    arr, pool, plen = table_array(table)
    n = len(table)
    offs = np.zeros(max(n, 1), np.int64)
    model.ctx.check(lib().mure_expand_patches_noalloc(model.h, _ptr(arr), n, _ptr(pool), plen, _ptr(out_dev),
                                                      int(out_dev.numel()), _ptr(offs)))
    return offs[:n]


def mure_check_descriptors(model, table=None, precision: str = "fp32"):
    """Host-side validation of a network description and (optionally) a mutant table,
    with no context and no device: (status, reason); status 0 = MURE_OK."""
    desc, keep = _model_desc(model, precision)
    arr, pool, plen = table_array(table) if table is not None else (None, None, 0)
    n = len(table) if table is not None else 0
    msg = C.create_string_buffer(512)
    st = lib().mure_check_descriptors(C.byref(desc), _ptr(arr) if n else None, n,
                                      _ptr(pool) if plen else None, plen, msg, 512)
    return int(st), msg.value.decode()
