"""Thin ctypes binding of libduo (include/duo.h): argument marshalling only.

Every step of the compute path runs in the library's CUDA kernels; PyTorch
only provides device memory and streams.  There is no fallback: if
``libduo.so`` is missing or cannot be loaded, :func:`load_library` raises.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libduo.so")

DUO_OK, DUO_EINVAL, DUO_ENOMEM, DUO_ECUDA, DUO_ERANGE, DUO_EFORMAT, DUO_ETIMEOUT = 0, -1, -2, -3, -4, -5, -6
DUO_FMT_IDX16, DUO_FMT_BITMASK, DUO_FMT_BITMASK_Q8, DUO_FMT_BITMASK_Q4 = 0, 1, 2, 3
FORMATS = {"idx16": DUO_FMT_IDX16, "bitmask": DUO_FMT_BITMASK, "cmb": DUO_FMT_BITMASK,
           "bitmask_q8": DUO_FMT_BITMASK_Q8, "bitmask_q4": DUO_FMT_BITMASK_Q4}

_lib = None


class DuoError(RuntimeError):
    def __init__(self, code: int, what: str):
        self.code = code
        super().__init__(f"{what}: {duo_strerror(code)} ({code})")


class _Info(ctypes.Structure):
    _fields_ = [("fmt", ctypes.c_int32), ("version", ctypes.c_int32), ("magic", ctypes.c_uint32),
                ("seg_rows", ctypes.c_int32), ("out", ctypes.c_int64), ("inp", ctypes.c_int64),
                ("nseg", ctypes.c_int64), ("nnz", ctypes.c_int64),
                ("index_dev", ctypes.c_void_p), ("index_bytes", ctypes.c_int64),
                ("aux_dev", ctypes.c_void_p), ("aux_bytes", ctypes.c_int64),
                ("data_dev", ctypes.c_void_p), ("data_bytes", ctypes.c_int64)]


class _CalibInfo(ctypes.Structure):
    """Mirror of duo_calib_info (include/duo_calib.h)."""
    _fields_ = [("k", ctypes.c_int64), ("m", ctypes.c_int64),
                ("perm_dev", ctypes.c_void_p), ("H_dev", ctypes.c_void_p), ("L_dev", ctypes.c_void_p),
                ("Q_dev", ctypes.c_void_p), ("U_dev", ctypes.c_void_p), ("D_dev", ctypes.c_void_p),
                ("a_dev", ctypes.c_void_p), ("b_dev", ctypes.c_void_p), ("c_dev", ctypes.c_void_p),
                ("col_dev", ctypes.c_void_p)]


def load_library(path: str | None = None):
    """Loads libduo.so (once).  Raises if it is missing: there is no
    CPU or PyTorch fallback for any entry point."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"libduo.so not built ({p}); run paper_2506_20194_gb300.build")
    lib = ctypes.CDLL(p)
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    lib.duo_pack.argtypes = [vp, i64, i64, i64, i32, vp, ctypes.POINTER(vp)]
    lib.duo_sparsify.argtypes = [vp, i64, i64, vp, vp, vp]
    lib.duo_spmspv.argtypes = [vp, vp, vp, vp, i64, vp, vp]
    lib.duo_spmspv_multi.argtypes = [ctypes.POINTER(vp), i32, vp, vp, vp, i64, ctypes.POINTER(vp), vp]
    lib.duo_sparsify_threshold.argtypes = [vp, i64, ctypes.c_uint16, vp, vp, vp, vp]
    lib.duo_spmspv_threshold.argtypes = [ctypes.POINTER(vp), i32, vp, ctypes.c_uint16, ctypes.POINTER(vp), vp]
    lib.duo_free.argtypes = [vp]
    lib.duo_packed_query.argtypes = [vp, ctypes.POINTER(_Info)]
    lib.duo_packed_export.argtypes = [vp, i32, vp, i64]
    lib.duo_pack_cmb_noalloc.argtypes = [vp, i64, i64, i64, vp, vp, i64, ctypes.POINTER(i64), vp]
    lib.duo_device_status.argtypes = [vp]
    lib.duo_packed_status.argtypes = [vp, vp]
    # internal, for the failure-detection test (not part of include/duo.h)
    lib.duo_test_spmspv_blocked.argtypes = [vp, vp, i64, vp, ctypes.c_uint64, vp]
    # internal, for the tensor-core GEMM's parity tests
    lib.duo_test_tc_gemm.argtypes = [i32, i32, i32, i32, i32, vp, i64, i64, i64, vp, i64, i64, i64, vp, i64, i64,
                                     i64, ctypes.c_float, ctypes.c_float, i32, i32, vp]
    # internal, for the CPU test of the launcher's run plan
    lib.duo_test_plan_runs.argtypes = [i32, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_float), i32,
                                       ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_int)]
    lib.duo_copy.argtypes = [vp, vp, i64, vp]
    lib.duo_calib_create.argtypes = [i64, i64, vp, ctypes.POINTER(vp)]
    lib.duo_calib_precompute.argtypes = [vp, vp, i64, ctypes.c_float, i32, vp]
    lib.duo_calib_status.argtypes = [vp, vp]
    lib.duo_calib_query.argtypes = [vp, ctypes.POINTER(_CalibInfo)]
    lib.duo_calib_export.argtypes = [vp, i32, vp, i64, vp]
    lib.duo_calib_score.argtypes = [vp, vp, i64, i64, vp, vp]
    lib.duo_calib_prune.argtypes = [vp, vp, i64, i64, i32, i32, vp, vp, vp]
    lib.duo_calib_free.argtypes = [vp]
    lib.duo_strerror.argtypes = [i32]
    lib.duo_abi_version.argtypes = []
    lib.duo_strerror.restype = ctypes.c_char_p
    for name in ("duo_pack", "duo_sparsify", "duo_spmspv", "duo_spmspv_multi", "duo_free",
                 "duo_packed_query", "duo_packed_export", "duo_device_status", "duo_abi_version",
                 "duo_pack_cmb_noalloc", "duo_sparsify_threshold", "duo_spmspv_threshold",
                 "duo_calib_create", "duo_calib_precompute", "duo_calib_status", "duo_calib_export",
                 "duo_calib_score", "duo_calib_free", "duo_calib_prune", "duo_copy", "duo_calib_query",
                 "duo_packed_status", "duo_test_spmspv_blocked", "duo_test_tc_gemm", "duo_test_plan_runs"):
        getattr(lib, name).restype = ctypes.c_int
    _lib = lib
    return lib


def duo_strerror(code: int) -> str:
    return load_library().duo_strerror(int(code)).decode()


def _stream_ptr(stream) -> int | None:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _ptr(t: torch.Tensor | None):
    return None if t is None else t.data_ptr()


def _check(rc: int, what: str):
    if rc != DUO_OK:
        raise DuoError(rc, what)


@dataclass
class PackedInfo:
    fmt: int
    version: int
    magic: int
    seg_rows: int
    out: int
    inp: int
    nseg: int
    nnz: int
    index_dev: int
    index_bytes: int
    aux_dev: int
    aux_bytes: int
    data_dev: int
    data_bytes: int


class Packed:
    """Owner of a duo_packed handle (freed by :meth:`free` or on collection)."""

    def __init__(self, handle: int, out: int, inp: int, fmt: int):
        self._h = handle
        self.out, self.inp, self.fmt = out, inp, fmt

    @property
    def handle(self) -> int:
        if not self._h:
            raise DuoError(DUO_EINVAL, "handle already freed")
        return self._h

    def query(self) -> PackedInfo:
        info = _Info()
        _check(load_library().duo_packed_query(self.handle, ctypes.byref(info)), "duo_packed_query")
        return PackedInfo(*[getattr(info, f[0]) or 0 for f in _Info._fields_])

    def free(self):
        if self._h:
            h, self._h = self._h, None
            _check(load_library().duo_free(h), "duo_free")

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def duo_pack(W: torch.Tensor, fmt="bitmask", stream=None) -> Packed:
    """Packs an O x I fp16 CUDA weight (pruned entries zero); see duo_pack in
    include/duo.h.  Row-major with unit column stride; any row stride."""
    if W.dtype != torch.float16 or W.dim() != 2 or not W.is_cuda:
        raise DuoError(DUO_EINVAL, "duo_pack needs a 2-D fp16 CUDA tensor")
    if W.stride(1) != 1:
        raise DuoError(DUO_EINVAL, "duo_pack needs unit column stride")
    f = FORMATS[fmt] if isinstance(fmt, str) else int(fmt)
    h = ctypes.c_void_p()
    O, I = W.shape
    _check(load_library().duo_pack(W.data_ptr(), O, I, W.stride(0), f, _stream_ptr(stream),
                                   ctypes.byref(h)), "duo_pack")
    return Packed(h.value, O, I, f)


def duo_sparsify(x: torch.Tensor, k: int, kept_idx: torch.Tensor | None = None,
                 kept_val: torch.Tensor | None = None, stream=None):
    """Kept channel ids (uint16 bits in an int16 tensor, ascending) and their
    fp16 values for the k largest |x| (§3)."""
    I = x.numel()
    if kept_idx is None:
        kept_idx = torch.empty(k, dtype=torch.int16, device=x.device)
    if kept_val is None:
        kept_val = torch.empty(k, dtype=torch.float16, device=x.device)
    _check(load_library().duo_sparsify(_ptr(x), I, int(k), _ptr(kept_idx), _ptr(kept_val),
                                       _stream_ptr(stream)), "duo_sparsify")
    return kept_idx, kept_val


def duo_spmspv(h: Packed, x: torch.Tensor | None, k: int, kept_idx=None, kept_val=None,
               y: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """y = W (x ⊙ m^x) (§3): fused selection when kept_idx/kept_val are None."""
    if y is None:
        dev = (x if x is not None else kept_idx).device
        y = torch.empty(h.out, dtype=torch.float32, device=dev)
    _check(load_library().duo_spmspv(h.handle, _ptr(x), _ptr(kept_idx), _ptr(kept_val), int(k),
                                     _ptr(y), _stream_ptr(stream)), "duo_spmspv")
    return y


def duo_spmspv_multi(hs, x: torch.Tensor | None, k: int, kept_idx=None, kept_val=None,
                     ys=None, stream=None):
    """n products sharing one sparse input (q/k/v, gate/up) in one launch."""
    n = len(hs)
    if ys is None:
        dev = (x if x is not None else kept_idx).device
        ys = [torch.empty(h.out, dtype=torch.float32, device=dev) for h in hs]
    harr = (ctypes.c_void_p * n)(*[h.handle for h in hs])
    yarr = (ctypes.c_void_p * n)(*[y.data_ptr() for y in ys])
    _check(load_library().duo_spmspv_multi(harr, n, _ptr(x), _ptr(kept_idx), _ptr(kept_val),
                                           int(k), yarr, _stream_ptr(stream)), "duo_spmspv_multi")
    return ys


def tau_bits(tau) -> int:
    """fp16 bit pattern of a threshold given as a number or an fp16 tensor."""
    if isinstance(tau, torch.Tensor):
        return int(tau.reshape(()).to(torch.float16).view(torch.int16).item()) & 0xFFFF
    return int(torch.tensor(float(tau), dtype=torch.float16).view(torch.int16).item()) & 0xFFFF


def duo_sparsify_threshold(x: torch.Tensor, tau, stream=None):
    """Channels with |x_j| > |tau| (§5, threshold mask), ascending: returns
    (kept_idx, kept_val, count) with room for every channel; the first
    ``count`` (a device int32 tensor) entries are valid."""
    I = x.numel()
    kept_idx = torch.empty(I, dtype=torch.int16, device=x.device)
    kept_val = torch.empty(I, dtype=torch.float16, device=x.device)
    count = torch.empty(1, dtype=torch.int32, device=x.device)
    _check(load_library().duo_sparsify_threshold(_ptr(x), I, tau_bits(tau), _ptr(kept_idx),
                                                 _ptr(kept_val), _ptr(count), _stream_ptr(stream)),
           "duo_sparsify_threshold")
    return kept_idx, kept_val, count


def duo_spmspv_threshold(hs, x: torch.Tensor, tau, ys=None, stream=None):
    """y_p = W_p (x ⊙ m^x) with the threshold mask |x_j| > |tau| computed in
    the launch, for n products sharing x (a list of handles, or one)."""
    if isinstance(hs, Packed):
        hs = [hs]
    n = len(hs)
    if ys is None:
        ys = [torch.empty(h.out, dtype=torch.float32, device=x.device) for h in hs]
    harr = (ctypes.c_void_p * n)(*[h.handle for h in hs])
    yarr = (ctypes.c_void_p * n)(*[y.data_ptr() for y in ys])
    _check(load_library().duo_spmspv_threshold(harr, n, _ptr(x), tau_bits(tau), yarr,
                                               _stream_ptr(stream)), "duo_spmspv_threshold")
    return ys


def duo_free(h: Packed):
    h.free()


def duo_device_status(stream=None) -> int:
    return load_library().duo_device_status(_stream_ptr(stream))


def duo_packed_status(h: Packed, stream=None) -> int:
    """Status of the launches whose first handle is h (read and cleared)."""
    return load_library().duo_packed_status(h.handle, _stream_ptr(stream))


def duo_copy(dst: torch.Tensor, src: torch.Tensor, stream=None):
    """dst <- src (same byte size, contiguous) by the library's SM copy
    kernel; either side may be a CUDA tensor or a pinned host tensor."""
    if not (dst.is_contiguous() and src.is_contiguous()):
        raise ValueError("duo_copy needs contiguous tensors")
    n = dst.numel() * dst.element_size()
    if src.numel() * src.element_size() != n:
        raise ValueError("duo_copy: sizes differ")
    _check(load_library().duo_copy(dst.data_ptr(), src.data_ptr(), n, _stream_ptr(stream)), "duo_copy")


def packed_bytes(h: Packed):
    """Copies a handle's index / aux / data buffers to host numpy uint8
    arrays through duo_packed_export (byte-level parity checks, saving)."""
    import numpy as np
    info = h.query()
    lib = load_library()
    out = []
    for which, n in ((0, info.index_bytes), (1, info.aux_bytes), (2, info.data_bytes)):
        buf = np.zeros(n, dtype=np.uint8)
        _check(lib.duo_packed_export(h.handle, which, buf.ctypes.data if n else None, n),
               "duo_packed_export")
        out.append(buf)
    return (info, *out)


def duo_pack_cmb_noalloc(W: torch.Tensor, off: torch.Tensor | None = None,
                         data: torch.Tensor | None = None, stream=None):
    """Bitmask packing into caller-owned buffers through the entry point that
    allocates nothing on the device (see duo_pack_cmb_noalloc in
    include/duo.h).  Missing buffers are allocated here, by the caller side,
    with PyTorch; returns (off int32 tensor, data uint8 tensor, data bytes)."""
    if W.dtype != torch.float16 or W.dim() != 2 or not W.is_cuda or W.stride(1) != 1:
        raise DuoError(DUO_EINVAL, "duo_pack_cmb_noalloc needs a 2-D fp16 CUDA tensor")
    O, I = W.shape
    S = (O + 1023) // 1024
    lib = load_library()
    if off is None:
        off = torch.empty(I * S + 1, dtype=torch.int32, device=W.device)
    nb = ctypes.c_int64(0)
    st = _stream_ptr(stream)
    if data is None:
        _check(lib.duo_pack_cmb_noalloc(W.data_ptr(), O, I, W.stride(0), off.data_ptr(), None, 0,
                                        ctypes.byref(nb), st), "duo_pack_cmb_noalloc")
        data = torch.empty(max(16, nb.value), dtype=torch.uint8, device=W.device)
    _check(lib.duo_pack_cmb_noalloc(W.data_ptr(), O, I, W.stride(0), off.data_ptr(), data.data_ptr(),
                                    data.numel(), ctypes.byref(nb), st), "duo_pack_cmb_noalloc")
    return off, data, nb.value


_CALIB_BUFS = {"perm": (0, torch.int32, 1), "H": (1, torch.float32, 2), "L": (2, torch.float32, 2),
               "Q": (3, torch.float32, 2), "U": (4, torch.float32, 2), "D": (5, torch.float32, 2),
               "a": (6, torch.float32, 1), "b": (7, torch.float32, 1), "c": (8, torch.float32, 1),
               "col": (9, torch.float32, 1)}


class Calib:
    """Context of the calibration precompute (§4.3, Algorithm 1) for k
    channels and m tokens; see include/duo_calib.h."""

    def __init__(self, k: int, m: int, stream=None):
        h = ctypes.c_void_p()
        _check(load_library().duo_calib_create(int(k), int(m), _stream_ptr(stream), ctypes.byref(h)),
               "duo_calib_create")
        self._h, self.k, self.m = h.value, int(k), int(m)

    def precompute(self, X: torch.Tensor, keep: int, damp: float = 0.1, act_order: bool = True,
                   stream=None):
        """X: m x k fp16 CUDA tensor, one row per token (the paper's X is k x m)."""
        if X.dtype != torch.float16 or tuple(X.shape) != (self.m, self.k) or not X.is_contiguous():
            raise DuoError(DUO_EINVAL, "precompute needs a contiguous m x k fp16 tensor")
        _check(load_library().duo_calib_precompute(self._h, X.data_ptr(), int(keep), float(damp),
                                                   1 if act_order else 0, _stream_ptr(stream)),
               "duo_calib_precompute")

    def status(self, stream=None) -> int:
        return load_library().duo_calib_status(self._h, _stream_ptr(stream))

    def query(self) -> dict:
        """duo_calib_query: k, m and the device addresses of the context's
        buffers (owned by the context; valid until the next precompute)."""
        info = _CalibInfo()
        _check(load_library().duo_calib_query(self._h, ctypes.byref(info)), "duo_calib_query")
        return {name: getattr(info, name) for name, _ in _CalibInfo._fields_}

    def get(self, name: str, stream=None) -> torch.Tensor:
        which, dt, nd = _CALIB_BUFS[name]
        shape = (self.k, self.k) if nd == 2 else (self.k,)
        out = torch.empty(shape, dtype=dt, device="cuda")
        _check(load_library().duo_calib_export(self._h, which, out.data_ptr(), out.numel() * 4,
                                               _stream_ptr(stream)), "duo_calib_export")
        return out

    def score(self, W: torch.Tensor, S: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        """S = W^2 (1 / L_pp^2 + a - b + 2 c), columns in the processing order."""
        if W.dtype != torch.float16 or W.dim() != 2 or W.shape[1] != self.k or W.stride(1) != 1:
            raise DuoError(DUO_EINVAL, "score needs an n x k fp16 tensor with unit column stride")
        if S is None:
            S = torch.empty(W.shape[0], self.k, dtype=torch.float32, device=W.device)
        _check(load_library().duo_calib_score(self._h, W.data_ptr(), W.shape[0], W.stride(0),
                                              S.data_ptr(), _stream_ptr(stream)), "duo_calib_score")
        return S

    def prune(self, W: torch.Tensor, pw_pct: int, block: int = 128, stream=None):
        """Algorithm 1's column sweep: returns (pruned fp32 n x k, keep uint8
        n x k), both in the original channel order."""
        if W.dtype != torch.float16 or W.dim() != 2 or W.shape[1] != self.k or W.stride(1) != 1:
            raise DuoError(DUO_EINVAL, "prune needs an n x k fp16 tensor with unit column stride")
        out = torch.empty(W.shape[0], self.k, dtype=torch.float32, device=W.device)
        keep = torch.empty(W.shape[0], self.k, dtype=torch.uint8, device=W.device)
        _check(load_library().duo_calib_prune(self._h, W.data_ptr(), W.shape[0], W.stride(0), int(pw_pct),
                                              int(block), out.data_ptr(), keep.data_ptr(),
                                              _stream_ptr(stream)), "duo_calib_prune")
        return out, keep

    def free(self):
        if self._h:
            h, self._h = self._h, None
            _check(load_library().duo_calib_free(h), "duo_calib_free")

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


class StepGraph:
    """A decode step of several dual-sparse products, captured once as a
    CUDA graph and replayed with one call: one host -> device copy of all the
    step's inputs, the products back to back, one device -> host copy of all
    outputs.  The two copies are the library's SM copy kernel (duo_copy) on
    the pinned buffers, not copy-engine nodes (about 4 us less per step).

    ``stages`` is a list of dicts: ``h`` (a Packed, or a list of up to 4
    sharing one input) and ``k`` (kept channels).  The object owns one pinned
    host buffer for the inputs and one for the outputs; ``x_host(i)`` and
    ``y_host(i, j)`` are views of them (fp16 input of stage i, fp32 output of
    its j-th product).  Write the next inputs into the x_host views before
    :meth:`run`; the outputs are in the y_host views once the stream has
    finished."""

    def __init__(self, stages, stream=None):
        self._stages = []
        xoff = yoff = 0
        for st in stages:
            hs = list(st["h"]) if isinstance(st["h"], (list, tuple)) else [st["h"]]
            I = hs[0].inp
            yo = []
            for h in hs:
                yo.append((yoff, h.out))
                yoff += (h.out + 3) // 4 * 4            # 16-byte aligned outputs
            self._stages.append((hs, int(st["k"]), xoff, I, yo))
            xoff += (I + 7) // 8 * 8                     # 16-byte aligned inputs
        self._xh = torch.zeros(max(xoff, 8), dtype=torch.float16).pin_memory()
        self._yh = torch.zeros(max(yoff, 4), dtype=torch.float32).pin_memory()
        self._xd = torch.zeros_like(self._xh, device="cuda")
        self._yd = torch.zeros_like(self._yh, device="cuda")
        s = torch.cuda.Stream() if stream is None else stream
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):   # one eager pass (library state, launch attributes)
            self._enqueue()
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            self._enqueue()

    def x_host(self, i):
        _, _, off, I, _ = self._stages[i]
        return self._xh[off:off + I]

    def y_host(self, i, j=0):
        off, O = self._stages[i][4][j]
        return self._yh[off:off + O]

    def _enqueue(self):
        duo_copy(self._xd, self._xh)
        for hs, k, xo, I, yo in self._stages:
            x = self._xd[xo:xo + I]
            ys = [self._yd[o:o + O] for o, O in yo]
            if len(hs) == 1:
                duo_spmspv(hs[0], x, k, y=ys[0])
            else:
                duo_spmspv_multi(hs, x, k, ys=ys)
        duo_copy(self._yh, self._yd)

    def run(self):
        self.graph.replay()
