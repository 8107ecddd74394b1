"""Python binding of libct, the carry-through checksum inference library.

Argument marshalling only: every step of inference, verification, fault
injection and re-execution runs in the library's CUDA kernels (see
``include/ct.h``).  The functions keep the C names.  Device buffers are
passed as PyTorch CUDA tensors (or raw integer addresses); PyTorch supplies
device memory and streams, nothing else.

Importing this package does not need a GPU; calling into the library does,
and there is no fallback: if ``_lib/libct.so`` is missing, every call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import List, Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libct.so")

CT_FP32, CT_FP16 = 0, 1
CT_OP_CONV, CT_OP_MAXPOOL, CT_OP_GAP, CT_OP_FC = 0, 1, 2, 3
CT_ROLE_CT, CT_ROLE_NONE, CT_ROLE_PASS, CT_ROLE_AUTO = 0, 1, 2, 3
CT_BUF_WEIGHT, CT_BUF_ACT = 0, 1
CT_DS_PASS, CT_DS_ZERO = 0, 1
CT_PROTECT_NONE, CT_PROTECT_WIDEN, CT_PROTECT_REPLACE = 0, 1, 2
CT_FLAG_SIMT_ONLY = 1
CT_FLAG_LAYERWISE = 2
FAM_TC, FAM_SIMT, FAM_FC, FAM_POOL, FAM_OTHER = 0, 1, 2, 3, 4

_STATUS = {0: "CT_OK", 1: "CT_EINVAL", 2: "CT_ENOMEM", 3: "CT_ECUDA", 4: "CT_ESTATE",
           5: "CT_ERANGE", 6: "CT_EUNSUPPORTED", 7: "CT_EDEVICE"}

# every exported symbol of include/ct.h
EXPORTS = ["ct_build", "ct_set_threshold", "ct_get_threshold", "ct_infer", "ct_inject",
           "ct_clear_faults", "ct_reexecute", "ct_infer_reexec", "ct_run_host", "ct_calibrate", "ct_buffer_count",
           "ct_buffer_info", "ct_profile_enable", "ct_profile_read", "ct_launches_per_infer", "ct_kernel_count",
           "ct_fi_threshold",
           "ct_copy_activation", "ct_device_error", "ct_destroy", "ct_strerror",
           "ct_reexecute_noalloc", "ct_campaign_batched", "ct_resolve_roles",
           "ct_reexecute_prepare", "ct_infer_batches", "ct_run_host_batches"]

CT_NOALLOC_SCRATCH_BYTES = 16 * 1024 * 1024


class CtError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        self.status = status
        super().__init__("%s: %s (%s)" % (what, _STATUS.get(status, status), _strerror(status)))


class LayerDesc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("op", "src", "dst", "res", "cin", "cout", "k", "stride", "pad", "role", "bn",
                 "relu", "final", "ct_shift", "groups")]


class ModelDesc(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("layers", ctypes.POINTER(LayerDesc)),
                ("in_c", ctypes.c_int32), ("in_h", ctypes.c_int32), ("in_w", ctypes.c_int32),
                ("n_classes", ctypes.c_int32), ("bn_eps", ctypes.c_double)]


class FaultDesc(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("layer", ctypes.c_int32), ("element", ctypes.c_int64),
                ("bit", ctypes.c_int32)]


class BuildOpts(ctypes.Structure):
    _fields_ = [("precision", ctypes.c_int32), ("protect", ctypes.c_int32),
                ("ds_mode", ctypes.c_int32), ("device", ctypes.c_int32),
                ("max_batch", ctypes.c_int32), ("flags", ctypes.c_uint32)]


_lib = None


def lib():
    """The loaded libct.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libct.so is not built (%s); run paper_2609_16742_gb300.build.build()"
                               % LIB_PATH)
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, i64, dbl = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        P = ctypes.POINTER
        sig = {
            "ct_build": [P(ModelDesc), P(ctypes.c_void_p), P(BuildOpts), P(vp)],
            "ct_set_threshold": [vp, dbl, dbl],
            "ct_get_threshold": [vp, P(dbl), P(dbl)],
            "ct_infer": [vp, vp, i32, vp, vp, vp, vp],
            "ct_inject": [vp, i32, i32, i64, i32],
            "ct_clear_faults": [vp],
            "ct_reexecute": [vp, vp, i32, vp, vp, vp, P(i32), vp],
            "ct_infer_reexec": [vp, vp, i32, vp, vp, vp, vp, i32, vp, vp, vp, P(i32), vp],
            "ct_reexecute_noalloc": [vp, vp, i32, vp, vp, vp, P(i32), vp],
            "ct_run_host": [vp, vp, i32, vp, vp, vp, P(i32), vp],
            "ct_calibrate": [vp, i64, dbl, P(dbl), P(dbl)],
            "ct_fi_threshold": [vp, vp, i64, dbl, dbl, P(dbl)],
            "ct_buffer_count": [vp, i32, P(i32)],
            "ct_buffer_info": [vp, i32, i32, P(i32), P(i32), P(i64), P(i32)],
            "ct_profile_enable": [vp, i32],
            "ct_profile_read": [vp, i32, P(i64), P(dbl), P(dbl)],
            "ct_launches_per_infer": [vp, P(i32)],
            "ct_kernel_count": [vp, P(i64)],
            "ct_copy_activation": [vp, i32, i32, vp, vp, P(i32), P(i32), P(i32), P(i32), P(i32), vp],
            "ct_device_error": [vp, P(ctypes.c_uint32)],
            "ct_campaign_batched": [vp, vp, i32, P(FaultDesc), i32, vp, vp, vp, vp],
            "ct_resolve_roles": [P(ModelDesc), P(i32)],
            "ct_reexecute_prepare": [vp, i32],
            "ct_infer_batches": [vp, i32, i32, P(vp), P(vp), P(vp), P(vp), P(i32), vp],
            "ct_run_host_batches": [vp, i32, i32, P(vp), P(vp), P(vp), P(vp), P(i32), vp],
        }
        for name, args in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = ctypes.c_int
        L.ct_destroy.argtypes = [vp]
        L.ct_destroy.restype = None
        L.ct_strerror.argtypes = [ctypes.c_int]
        L.ct_strerror.restype = ctypes.c_char_p
        _lib = L
    return _lib


def _strerror(s: int) -> str:
    try:
        return lib().ct_strerror(int(s)).decode()
    except Exception:
        return "?"


def _check(s: int, what: str):
    if s != 0:
        raise CtError(s, what)


def _ptr(t) -> Optional[int]:
    """Device or host address of a torch tensor / numpy array / int / None."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


_OPS = {"conv": CT_OP_CONV, "maxpool": CT_OP_MAXPOOL, "gap": CT_OP_GAP, "fc": CT_OP_FC}
_ROLES = {"ct": CT_ROLE_CT, "none": CT_ROLE_NONE, "pass": CT_ROLE_PASS, "auto": CT_ROLE_AUTO}
_ROLE_NAMES = {v: k for k, v in _ROLES.items()}


class Model:
    """Handle of a built model (owns the C ct_model)."""

    def __init__(self, handle: int, n_classes: int, in_shape, precision: str, protect: bool,
                 max_batch: int):
        self.handle = ctypes.c_void_p(handle)
        self.n_classes = n_classes
        self.in_shape = tuple(in_shape)
        self.precision = precision
        self.protect = protect
        self.max_batch = max_batch

    def close(self):
        if self.handle:
            lib().ct_destroy(self.handle)
            self.handle = ctypes.c_void_p(0)

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _layer_descs(layers: Sequence):
    n = len(layers)
    arr = (LayerDesc * n)()
    for i, L in enumerate(layers):
        arr[i] = LayerDesc(_OPS[L.op], L.src, L.dst, L.res, L.cin, L.cout, L.k, L.stride, L.pad,
                           _ROLES.get(L.ct, CT_ROLE_NONE), int(L.bn), int(L.relu), int(L.final),
                           int(L.ct_shift), int(getattr(L, "groups", 1)))
    return arr


def ct_resolve_roles(layers: Sequence, in_shape, n_classes: int) -> List[Optional[str]]:
    """Sec. II-A residual rule as the library applies it: the effective role
    of every convolution ("ct", "none", "pass"; "auto" resolved), None for
    other layers.  Raises CtError (CT_EINVAL) when a "ct" role breaks the rule."""
    arr = _layer_descs(layers)
    desc = ModelDesc(len(layers), arr, in_shape[0], in_shape[1], in_shape[2], n_classes, 1e-5)
    out = (ctypes.c_int32 * len(layers))()
    _check(lib().ct_resolve_roles(ctypes.byref(desc), out), "ct_resolve_roles")
    return [None if r < 0 else _ROLE_NAMES[r] for r in out]


def ct_build(layers: Sequence, params: Sequence[dict], in_shape, n_classes: int,
             precision: str = "fp32", protect: bool = True, ds_mode: str = "pass",
             device: int = 0, max_batch: int = 64, simt_only: bool = False,
             bn_eps: float = 1e-5, replace: bool = False, layerwise: bool = False) -> Model:
    """Build a model from synth-style layers and float32 parameter dicts.

    protect=True adds the carry-through filters as extra channels (widened);
    replace=True builds the paper's prune-and-replace construction instead;
    layerwise=True keeps one kernel per layer: for the LeNet-5 shape, and for
    1x1 shortcuts that would otherwise run in their block's first launch."""
    n = len(layers)
    arr = _layer_descs(layers)
    keep = []
    wp = (ctypes.c_void_p * (6 * n))()
    for i, (L, p) in enumerate(zip(layers, params)):
        for j, key in enumerate(("w", "b", "gamma", "beta", "mean", "var")):
            if key in p:
                a = np.ascontiguousarray(p[key], dtype=np.float32)
                keep.append(a)
                wp[6 * i + j] = a.ctypes.data
    desc = ModelDesc(n, arr, in_shape[0], in_shape[1], in_shape[2], n_classes, bn_eps)
    mode = CT_PROTECT_REPLACE if replace else (CT_PROTECT_WIDEN if protect else CT_PROTECT_NONE)
    opts = BuildOpts(CT_FP16 if precision == "fp16" else CT_FP32, mode,
                     CT_DS_ZERO if ds_mode == "zero" else CT_DS_PASS, device, max_batch,
                     (CT_FLAG_SIMT_ONLY if simt_only else 0) | (CT_FLAG_LAYERWISE if layerwise else 0))
    h = ctypes.c_void_p()
    _check(lib().ct_build(ctypes.byref(desc), wp, ctypes.byref(opts), ctypes.byref(h)), "ct_build")
    return Model(h.value, n_classes, in_shape, precision, protect or replace, max_batch)


def ct_build_workload(wl, params=None, **kw) -> Model:
    import synth
    if params is None:
        params = synth.make_params(wl.layers, wl.seed)
    kw.setdefault("precision", wl.precision)
    kw.setdefault("max_batch", wl.batch)
    kw.setdefault("bn_eps", wl.bn_eps)
    return ct_build(wl.layers, params, wl.in_shape, wl.n_classes, **kw)


def ct_set_threshold(m: Model, reference: float, tau: float):
    _check(lib().ct_set_threshold(m.handle, reference, tau), "ct_set_threshold")


def ct_get_threshold(m: Model):
    r, t = ctypes.c_double(), ctypes.c_double()
    _check(lib().ct_get_threshold(m.handle, ctypes.byref(r), ctypes.byref(t)), "ct_get_threshold")
    return r.value, t.value


def ct_infer(m: Model, input_dev, batch: int, logits_dev, S_dev=None, flag_dev=None, stream=None):
    _check(lib().ct_infer(m.handle, _ptr(input_dev), batch, _ptr(logits_dev), _ptr(S_dev),
                          _ptr(flag_dev), _stream(stream)), "ct_infer")


def ct_inject(m: Model, kind: int, layer: int, element: int, bit: int):
    _check(lib().ct_inject(m.handle, kind, layer, element, bit), "ct_inject")


def ct_clear_faults(m: Model):
    _check(lib().ct_clear_faults(m.handle), "ct_clear_faults")


def ct_reexecute(m: Model, input_dev, batch: int, flag_dev, logits_dev, S_dev=None,
                 stream=None) -> int:
    n = ctypes.c_int32()
    _check(lib().ct_reexecute(m.handle, _ptr(input_dev), batch, _ptr(flag_dev), _ptr(logits_dev),
                              _ptr(S_dev), ctypes.byref(n), _stream(stream)), "ct_reexecute")
    return n.value


def ct_reexecute_prepare(m: Model, max_images: int):
    """Capture the re-execution graphs of every padded size up to max_images."""
    _check(lib().ct_reexecute_prepare(m.handle, max_images), "ct_reexecute_prepare")


def _ptr_array(items):
    """ctypes array of addresses (None entries stay NULL), or None for None."""
    if items is None:
        return None
    return (ctypes.c_void_p * max(len(items), 1))(*[_ptr(t) for t in items])


def ct_infer_batches(m: Model, inputs_dev, batch: int, logits_dev, S_dev, flag_dev, stream=None) -> int:
    """Inference of a list of device-resident batches with each batch's
    flagged images re-run two batches later (Sec. II-B); returns the images
    re-run.  Each argument is a list with one device tensor per batch."""
    n = ctypes.c_int32()
    _check(lib().ct_infer_batches(m.handle, len(inputs_dev), batch, _ptr_array(inputs_dev), _ptr_array(logits_dev),
                                  _ptr_array(S_dev), _ptr_array(flag_dev), ctypes.byref(n), _stream(stream)),
           "ct_infer_batches")
    return n.value


def ct_run_host_batches(m: Model, inputs_host, batch: int, logits_host, S_host=None, flag_host=None,
                        stream=None) -> int:
    """ct_infer_batches for host buffers (numpy arrays or pinned CPU tensors):
    input copies and result copies overlap the device's work."""
    n = ctypes.c_int32()
    _check(lib().ct_run_host_batches(m.handle, len(inputs_host), batch, _ptr_array(inputs_host),
                                     _ptr_array(logits_host), _ptr_array(S_host), _ptr_array(flag_host),
                                     ctypes.byref(n), _stream(stream)), "ct_run_host_batches")
    return n.value


def ct_infer_reexec(m: Model, input_dev, batch: int, logits_dev, S_dev=None, flag_dev=None,
                    prev_input_dev=None, prev_batch: int = 0, prev_flag_dev=None, prev_logits_dev=None,
                    prev_S_dev=None, stream=None) -> int:
    """ct_infer of a new batch that re-executes the previous batch's flagged
    images as extra rows of the same inference; returns how many were re-run."""
    n = ctypes.c_int32()
    _check(lib().ct_infer_reexec(m.handle, _ptr(input_dev), batch, _ptr(logits_dev), _ptr(S_dev), _ptr(flag_dev),
                                 _ptr(prev_input_dev), prev_batch, _ptr(prev_flag_dev), _ptr(prev_logits_dev),
                                 _ptr(prev_S_dev), ctypes.byref(n), _stream(stream)), "ct_infer_reexec")
    return n.value


def ct_campaign_batched(m: Model, input_dev, batch: int, faults, S_dev, top1_dev, flag_dev, stream=None):
    """Many faults in one launch.  faults: rows (kind, layer, element, bit);
    outputs [n_faults, batch] device tensors (float32, int32, uint8)."""
    f = np.asarray(faults, dtype=np.int64).reshape(-1, 4)
    arr = (FaultDesc * max(len(f), 1))()
    for i, (kind, layer, el, bit) in enumerate(f.tolist()):
        arr[i] = FaultDesc(kind, layer, el, bit)
    _check(lib().ct_campaign_batched(m.handle, _ptr(input_dev), batch, arr, len(f), _ptr(S_dev), _ptr(top1_dev),
                                     _ptr(flag_dev), _stream(stream)), "ct_campaign_batched")


def ct_reexecute_noalloc(m: Model, input_dev, batch: int, flag_dev, logits_dev, S_dev=None,
                         stream=None) -> int:
    """ct_reexecute without allocation: its scratch is a static device array."""
    n = ctypes.c_int32()
    _check(lib().ct_reexecute_noalloc(m.handle, _ptr(input_dev), batch, _ptr(flag_dev),
                                      _ptr(logits_dev), _ptr(S_dev), ctypes.byref(n),
                                      _stream(stream)), "ct_reexecute_noalloc")
    return n.value


def ct_run_host(m: Model, input_host: np.ndarray, logits_host: np.ndarray, S_host=None,
                flag_host=None, stream=None) -> int:
    assert input_host.dtype == np.float32 and input_host.flags.c_contiguous
    n = ctypes.c_int32()
    _check(lib().ct_run_host(m.handle, _ptr(input_host), input_host.shape[0], _ptr(logits_host),
                             _ptr(S_host), _ptr(flag_host), ctypes.byref(n), _stream(stream)),
           "ct_run_host")
    return n.value


def ct_calibrate(S_host: np.ndarray, alpha: float):
    S = np.ascontiguousarray(S_host, dtype=np.float32)
    r, t = ctypes.c_double(), ctypes.c_double()
    _check(lib().ct_calibrate(S.ctypes.data, S.size, alpha, ctypes.byref(r), ctypes.byref(t)),
           "ct_calibrate")
    return r.value, t.value


def ct_fi_threshold(S_host: np.ndarray, critical: np.ndarray, reference: float, alpha: float) -> float:
    """Sec. II-C FI-based threshold from campaign trials (S, critical)."""
    S = np.ascontiguousarray(S_host, dtype=np.float32)
    c = np.ascontiguousarray(critical, dtype=np.uint8)
    if S.shape != c.shape:
        raise ValueError("S and critical must have the same shape")
    t = ctypes.c_double()
    _check(lib().ct_fi_threshold(S.ctypes.data, c.ctypes.data, S.size, reference, alpha, ctypes.byref(t)),
           "ct_fi_threshold")
    return t.value


def ct_buffers(m: Model, batch: int) -> List[tuple]:
    """[(kind, layer, n_elements, bits)] from ct_buffer_count / ct_buffer_info."""
    n = ctypes.c_int32()
    _check(lib().ct_buffer_count(m.handle, batch, ctypes.byref(n)), "ct_buffer_count")
    out = []
    for i in range(n.value):
        k, l, b = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
        e = ctypes.c_int64()
        _check(lib().ct_buffer_info(m.handle, batch, i, ctypes.byref(k), ctypes.byref(l),
                                    ctypes.byref(e), ctypes.byref(b)), "ct_buffer_info")
        out.append((k.value, l.value, e.value, b.value))
    return out


def ct_profile_enable(m: Model, on: bool = True):
    _check(lib().ct_profile_enable(m.handle, int(on)), "ct_profile_enable")


def ct_profile_read(m: Model, family: int):
    n, ms, fl = ctypes.c_int64(), ctypes.c_double(), ctypes.c_double()
    _check(lib().ct_profile_read(m.handle, family, ctypes.byref(n), ctypes.byref(ms),
                                 ctypes.byref(fl)), "ct_profile_read")
    return n.value, ms.value, fl.value


def ct_kernel_count(m: Model) -> int:
    """Library kernels launched for m since the previous call (then reset)."""
    n = ctypes.c_int64()
    _check(lib().ct_kernel_count(m.handle, ctypes.byref(n)), "ct_kernel_count")
    return n.value


def ct_launches_per_infer(m: Model) -> int:
    n = ctypes.c_int32()
    _check(lib().ct_launches_per_infer(m.handle, ctypes.byref(n)), "ct_launches_per_infer")
    return n.value


def ct_copy_activation(m: Model, slot: int, batch: int, stream=None):
    """(data, cs) of a stored slot as float64 arrays: data [batch, C, H, W],
    cs [batch, H, W] or None."""
    C, H, W, hc, eb = (ctypes.c_int32() for _ in range(5))
    _check(lib().ct_copy_activation(m.handle, slot, batch, None, None, ctypes.byref(C),
                                    ctypes.byref(H), ctypes.byref(W), ctypes.byref(hc),
                                    ctypes.byref(eb), _stream(stream)), "ct_copy_activation")
    dt = np.float32 if eb.value == 4 else np.float16
    data = np.empty((batch, H.value, W.value, C.value), dt)
    cs = np.empty((batch, H.value, W.value), dt) if hc.value else None
    _check(lib().ct_copy_activation(m.handle, slot, batch, data.ctypes.data,
                                    None if cs is None else cs.ctypes.data, None, None, None,
                                    None, None, _stream(stream)), "ct_copy_activation")
    data = data.astype(np.float64).transpose(0, 3, 1, 2)
    return data, (None if cs is None else cs.astype(np.float64))


def ct_device_error(m: Model) -> int:
    c = ctypes.c_uint32()
    _check(lib().ct_device_error(m.handle, ctypes.byref(c)), "ct_device_error")
    return c.value


def ct_destroy(m: Model):
    m.close()
