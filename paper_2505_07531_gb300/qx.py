"""Python binding of libqx.so (ctypes): argument marshalling only.

Every computation runs in the library's CUDA kernels.  PyTorch supplies device
memory and the current CUDA stream; tensors are passed as raw pointers.  If
the library has not been built, importing this module raises: there is no CPU
or PyTorch fallback.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "lib", "libqx.so")

UNIFORM, LUT, Q4X = 0, 1, 2
F16, F32 = 0, 1
GEMV_PDL = 1
GEMV_SEPARATE = 2  # fused calls: one launch per group, each balanced with the workspace
GEMM_PDL = 1

STATUS = {
    0: "QX_OK",
    1: "QX_ERR_INVALID_ARG",
    2: "QX_ERR_UNSUPPORTED",
    3: "QX_ERR_ALIGNMENT",
    4: "QX_ERR_CUDA",
    5: "QX_ERR_TIMEOUT",
    6: "QX_ERR_NONFINITE",
}


class QxError(RuntimeError):
    """A non-zero qx_status returned by the library."""

    def __init__(self, code: int, where: str):
        self.code = code
        self.name = STATUS.get(code, str(code))
        detail = _lib().qx_status_string(code).decode()
        if code == 4:
            detail += ": " + _lib().qx_last_error_string().decode()
        super().__init__(f"{where}: {self.name} ({detail})")


class _Recipe(ctypes.Structure):
    _fields_ = [("bits", ctypes.c_int32), ("group_size", ctypes.c_int32),
                ("kind", ctypes.c_int32), ("lloyd_iters", ctypes.c_int32)]


class _Sizes(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_uint64), ("scales", ctypes.c_uint64),
                ("zeros", ctypes.c_uint64), ("luts", ctypes.c_uint64)]


class _Packed(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int64), ("k", ctypes.c_int64), ("recipe", _Recipe),
                ("codes", ctypes.c_void_p), ("scales", ctypes.c_void_p),
                ("zeros", ctypes.c_void_p), ("luts", ctypes.c_void_p)]


class _GemvGroup(ctypes.Structure):
    _fields_ = [("mats", ctypes.POINTER(_Packed)), ("count", ctypes.c_int32),
                ("x", ctypes.POINTER(ctypes.c_void_p)), ("y", ctypes.POINTER(ctypes.c_void_p))]


class _Copy(ctypes.Structure):
    _fields_ = [("dst", ctypes.c_void_p), ("src", ctypes.c_void_p), ("bytes", ctypes.c_size_t)]


class _Q4x(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int64), ("k", ctypes.c_int64), ("codes", ctypes.c_void_p),
                ("scales", ctypes.c_void_p), ("books", ctypes.c_void_p), ("codebooks", ctypes.c_void_p)]


class _Q4xSizes(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_uint64), ("scales", ctypes.c_uint64),
                ("books", ctypes.c_uint64), ("codebooks", ctypes.c_uint64)]


_LIB = None


def library_path() -> str:
    return _LIB_PATH


def _lib():
    global _LIB
    if _LIB is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(
                f"{_LIB_PATH} is missing: build it with paper_2505_07531_gb300.build.build_library() "
                "(there is no fallback path)")
        lib = ctypes.CDLL(_LIB_PATH)
        P, I32, I64, VP = ctypes.POINTER, ctypes.c_int32, ctypes.c_int64, ctypes.c_void_p
        lib.qx_packed_size.argtypes = [I64, I64, P(_Recipe), P(_Sizes)]
        lib.qx_quantize.argtypes = [VP, I64, I64, P(_Recipe), P(_Packed), VP]
        lib.qx_dequant.argtypes = [P(_Packed), VP, VP]
        lib.qx_gemv.argtypes = [P(_Packed), VP, I32, VP, I32, VP]
        lib.qx_gemm.argtypes = [P(_Packed), VP, I64, VP, VP]
        lib.qx_gemm_splitk_workspace.argtypes = [I64, I64, I64, P(_Recipe), P(ctypes.c_size_t)]
        lib.qx_gemm_splitk.argtypes = [P(_Packed), VP, I64, VP, VP, ctypes.c_size_t, I32, VP]
        lib.qx_gemm_splitk_plan.argtypes = [I64, I64, I64, I32, P(I32), P(I32), P(ctypes.c_size_t)]
        lib.qx_gemm_splitk_noalloc.argtypes = [P(_Packed), VP, I64, VP, VP]
        lib.qx_quantize_act.argtypes = [VP, I32, I64, VP, VP, VP]
        lib.qx_gemv_a8.argtypes = [P(_Packed), VP, VP, I32, VP, I32, VP]
        lib.qx_dequant_act.argtypes = [VP, VP, I64, I64, VP, VP]
        lib.qx_select_workspace.argtypes = [I64, I64, P(_Recipe), I32, P(ctypes.c_size_t)]
        lib.qx_select_recipe.argtypes = [VP, I64, I64, P(_Recipe), I32, ctypes.c_double, VP, ctypes.c_size_t,
                                         P(I32), P(ctypes.c_uint64), P(ctypes.c_double), VP]
        lib.qx_gemv_multi.argtypes = [P(_Packed), I32, P(VP), I32, P(VP), I32, I32, VP]
        lib.qx_gemv_chain.argtypes = [P(_GemvGroup), I32, I32, I32, I32, VP]
        lib.qx_decode_step.argtypes = [P(_Copy), I32, P(_GemvGroup), I32, I32, I32, I32, P(_Copy), I32, I32, VP]
        lib.qx_gemv_fused_workspace.argtypes = [P(ctypes.c_size_t)]
        lib.qx_gemv_fused.argtypes = [P(_GemvGroup), I32, I32, I32, I32, VP, ctypes.c_size_t, VP]
        lib.qx_decode_step_fused.argtypes = [P(_Copy), I32, P(_GemvGroup), I32, I32, I32, I32, VP, ctypes.c_size_t,
                                             P(_Copy), I32, I32, VP]
        lib.qx_q4x_size.argtypes = [I64, I64, P(_Q4xSizes)]
        lib.qx_q4x_workspace.argtypes = [I64, I64, P(ctypes.c_size_t)]
        lib.qx_q4x_quantize.argtypes = [VP, I32, P(_Q4x), VP, ctypes.c_size_t, VP]
        lib.qx_q4x_dequant.argtypes = [P(_Q4x), VP, VP]
        lib.qx_q4x_gemv.argtypes = [P(_Q4x), VP, I32, VP, I32, VP]
        lib.qx_q4x_gemv_multi.argtypes = [P(_Q4x), I32, P(VP), I32, P(VP), I32, VP]
        lib.qx_q4x_gemm.argtypes = [P(_Q4x), VP, I64, VP, VP]
        lib.qx_q4x_gemm_splitk_workspace.argtypes = [I64, I64, I64, P(ctypes.c_size_t)]
        lib.qx_q4x_gemm_splitk.argtypes = [P(_Q4x), VP, I64, VP, VP, ctypes.c_size_t, I32, VP]
        lib.qx_selftest_wait_timeout.argtypes = [I32, VP]
        lib.qx_get_device_status.argtypes = [VP]
        lib.qx_status_string.argtypes = [ctypes.c_int]
        lib.qx_status_string.restype = ctypes.c_char_p
        lib.qx_version.argtypes = []
        lib.qx_last_error_string.argtypes = []
        lib.qx_last_error_string.restype = ctypes.c_char_p
        for fn in ("qx_packed_size", "qx_quantize", "qx_dequant", "qx_gemv", "qx_gemv_multi", "qx_gemv_chain", "qx_decode_step", "qx_gemv_fused_workspace", "qx_gemv_fused",
                   "qx_decode_step_fused", "qx_gemm",
                   "qx_gemm_splitk_workspace", "qx_gemm_splitk", "qx_gemm_splitk_noalloc", "qx_gemm_splitk_plan",
                   "qx_select_workspace", "qx_select_recipe", "qx_quantize_act", "qx_dequant_act", "qx_gemv_a8",
                   "qx_q4x_size", "qx_q4x_workspace", "qx_q4x_quantize", "qx_q4x_dequant", "qx_q4x_gemv", "qx_q4x_gemv_multi", "qx_q4x_gemm", "qx_q4x_gemm_splitk_workspace",
                   "qx_q4x_gemm_splitk", "qx_selftest_wait_timeout",
                   "qx_get_device_status", "qx_version"):
            getattr(lib, fn).restype = ctypes.c_int
        _LIB = lib
    return _LIB


def _check(code: int, where: str):
    if code != 0:
        raise QxError(code, where)


@dataclass(frozen=True)
class Recipe:
    """Per-matrix recipe: bit-width, group size along k, uniform (0) or LUT (1);
    Q4X (2, bits 4, group 64) only as a select_recipe candidate."""

    bits: int
    group_size: int
    kind: int = UNIFORM
    lloyd_iters: int = 25

    def c(self) -> _Recipe:
        return _Recipe(self.bits, self.group_size, self.kind, self.lloyd_iters)


def packed_size(n: int, k: int, recipe: Recipe) -> dict:
    """Byte sizes of the packed buffers (host-only call)."""
    s = _Sizes()
    r = recipe.c()
    _check(_lib().qx_packed_size(n, k, ctypes.byref(r), ctypes.byref(s)), "qx_packed_size")
    return {"codes": s.codes, "scales": s.scales, "zeros": s.zeros, "luts": s.luts}


_RAW_STREAM = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _stream(dev) -> ctypes.c_void_p:
    """The current CUDA stream of device `dev` (a torch.device or an index)."""
    idx = dev.index if isinstance(dev, torch.device) else dev
    if idx is None:
        idx = torch.cuda.current_device()
    if _RAW_STREAM is not None:  # the same handle, without building a Stream object
        return ctypes.c_void_p(_RAW_STREAM(idx))
    return ctypes.c_void_p(torch.cuda.current_stream(idx).cuda_stream)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


class PackedMatrix:
    """Packed weights of one n x k matrix, held in torch device tensors."""

    def __init__(self, n, k, recipe, codes, scales=None, zeros=None, luts=None):
        self.n, self.k, self.recipe = int(n), int(k), recipe
        self.codes, self.scales, self.zeros, self.luts = codes, scales, zeros, luts
        self._c_key, self._c_struct = None, None

    @classmethod
    def empty(cls, n: int, k: int, recipe: Recipe, device) -> "PackedMatrix":
        sz = packed_size(n, k, recipe)
        u8 = dict(dtype=torch.uint8, device=device)
        codes = torch.empty(sz["codes"], **u8)
        scales = torch.empty(sz["scales"] // 2, dtype=torch.float16, device=device) if sz["scales"] else None
        zeros = torch.empty(sz["zeros"], **u8) if sz["zeros"] else None
        luts = torch.empty(sz["luts"] // 2, dtype=torch.float16, device=device) if sz["luts"] else None
        return cls(n, k, recipe, codes, scales, zeros, luts)

    @property
    def device(self):
        return self.codes.device

    def nbytes(self) -> int:
        return sum(t.numel() * t.element_size() for t in (self.codes, self.scales, self.zeros, self.luts)
                   if t is not None)

    def c(self) -> _Packed:
        # the ctypes struct is kept while the buffers stay the same (decode calls
        # it for every matrix of every step)
        key = tuple(None if t is None else t.data_ptr() for t in (self.codes, self.scales, self.zeros, self.luts))
        if key != self._c_key:
            self._c_struct = _Packed(self.n, self.k, self.recipe.c(), *key)
            self._c_key = key
        return self._c_struct

    def to_numpy(self) -> dict:
        """Host copies in the oracle's array shapes (for tests)."""
        G = self.k // self.recipe.group_size
        out = {"codes": self.codes.cpu().numpy().reshape(self.n, -1), "scales": None, "zeros": None, "luts": None}
        if self.scales is not None:
            out["scales"] = self.scales.cpu().numpy().reshape(self.n, G)
            out["zeros"] = self.zeros.cpu().numpy().reshape(self.n, -1)
        if self.luts is not None:
            out["luts"] = self.luts.cpu().numpy().reshape(self.n, G, 1 << self.recipe.bits)
        return out


def _on_device(t: torch.Tensor) -> bool:
    """Whether the library may take t's memory as device memory."""
    return t.is_cuda


def _dev_tensor(t: torch.Tensor, name: str, dtype=torch.float16):
    if not _on_device(t):
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def quantize(W: torch.Tensor, recipe: Recipe, out: PackedMatrix | None = None) -> PackedMatrix:
    """Quantize and pack fp16 W [n][k] on its device (qx_quantize)."""
    _dev_tensor(W, "W")
    n, k = W.shape
    P = out if out is not None else PackedMatrix.empty(n, k, recipe, W.device)
    r = recipe.c()
    pc = P.c()
    _check(_lib().qx_quantize(_ptr(W), n, k, ctypes.byref(r), ctypes.byref(pc), _stream(W.device)),
           "qx_quantize")
    return P


def dequant(P: PackedMatrix, out: torch.Tensor | None = None) -> torch.Tensor:
    """fp16 W_hat [n][k] (qx_dequant)."""
    W = out if out is not None else torch.empty((P.n, P.k), dtype=torch.float16, device=P.device)
    _dev_tensor(W, "out")
    pc = P.c()
    _check(_lib().qx_dequant(ctypes.byref(pc), _ptr(W), _stream(P.device)), "qx_dequant")
    return W


def gemv(P: PackedMatrix, x: torch.Tensor, out: torch.Tensor | None = None,
         out_dtype=torch.float16) -> torch.Tensor:
    """Decode y = x W_hat^T for x [batch][k] (qx_gemv); returns [batch][n]."""
    _dev_tensor(x, "x")
    x2 = x.view(-1, P.k)
    b = x2.shape[0]
    dt = out.dtype if out is not None else out_dtype
    y = out if out is not None else torch.empty((b, P.n), dtype=dt, device=x.device)
    _dev_tensor(y, "out", dt)
    code = F32 if dt == torch.float32 else F16
    pc = P.c()
    _check(_lib().qx_gemv(ctypes.byref(pc), _ptr(x2), b, _ptr(y), code, _stream(x.device)), "qx_gemv")
    return y


def gemv_multi(mats, xs, outs=None, out_dtype=torch.float16, pdl: bool = False):
    """Several decode matmuls in one launch (qx_gemv_multi); returns the outputs.

    ``mats`` share bits and kind; ``xs[i]`` is [batch][k_i].  ``pdl`` lets the
    kernel start while the previous kernel in the stream runs: set it only when
    that kernel does not write these weights.
    """
    mats, xs = list(mats), list(xs)
    if len(mats) != len(xs) or not mats:
        raise ValueError("need one x per matrix")
    for x in xs:
        _dev_tensor(x, "x")
    b = xs[0].numel() // mats[0].k
    dt = outs[0].dtype if outs is not None else out_dtype
    ys = list(outs) if outs is not None else [torch.empty((b, P.n), dtype=dt, device=xs[0].device) for P in mats]
    for y in ys:
        _dev_tensor(y, "out", dt)
    arr = (_Packed * len(mats))(*[P.c() for P in mats])
    xp = (ctypes.c_void_p * len(xs))(*[x.data_ptr() for x in xs])
    yp = (ctypes.c_void_p * len(ys))(*[y.data_ptr() for y in ys])
    code = F32 if dt == torch.float32 else F16
    _check(_lib().qx_gemv_multi(arr, len(mats), xp, b, yp, code, GEMV_PDL if pdl else 0, _stream(xs[0].get_device())),
           "qx_gemv_multi")
    return ys


class GemvChain:
    """A decode step as one qx_gemv_chain call.  `groups` lists (matrices, xs,
    outs) triples, each the arguments of one gemv_multi (same batch and output
    dtype throughout); the ctypes arguments are built here once, so calling
    the object costs one library call.  Build a new chain if any of the
    tensors is replaced.  With `fused`, the groups run as ONE persistent launch
    (qx_gemv_fused: its CTAs balanced slice by slice, so the results are within
    fp32 rounding of the chain's), on a workspace the object owns: do not call
    one fused object on two streams at the same time.  With `separate` (which
    implies the workspace) every group is a balanced launch of its own."""

    def __init__(self, groups, pdl: bool = True, fused: bool = False, separate: bool = False):
        fused = fused or separate
        self._keep, built = [], []
        batch, dt, dev = None, None, None
        for mats, xs, outs in groups:
            mats, xs, outs = list(mats), list(xs), list(outs)
            if not (len(mats) == len(xs) == len(outs)) or not 1 <= len(mats) <= 8:
                raise ValueError("each group: 1..8 matrices, one x and one output per matrix")
            for P, x, y in zip(mats, xs, outs):
                x2 = x.view(-1, P.k)
                _dev_tensor(x2, "x")
                b = x2.shape[0]
                batch = b if batch is None else batch
                dt = y.dtype if dt is None else dt
                dev = x.device if dev is None else dev
                if b != batch or y.dtype != dt or tuple(y.shape) != (b, P.n):
                    raise ValueError("every group must share the batch and the output dtype")
                _dev_tensor(y, "out", dt)
            cnt = len(mats)
            pa = (_Packed * cnt)(*[P.c() for P in mats])
            xa = (ctypes.c_void_p * cnt)(*[x.data_ptr() for x in xs])
            ya = (ctypes.c_void_p * cnt)(*[y.data_ptr() for y in outs])
            self._keep += [pa, xa, ya, mats, xs, outs]
            built.append(_GemvGroup(ctypes.cast(pa, ctypes.POINTER(_Packed)), cnt,
                                    ctypes.cast(xa, ctypes.POINTER(ctypes.c_void_p)),
                                    ctypes.cast(ya, ctypes.POINTER(ctypes.c_void_p))))
        if not built:
            raise ValueError("no groups")
        self._groups = (_GemvGroup * len(built))(*built)
        self._args = (self._groups, len(built), batch, F32 if dt == torch.float32 else F16,
                      (GEMV_PDL if pdl else 0) | (GEMV_SEPARATE if separate else 0))
        self._dev = dev
        self._ws = None
        if fused:
            nbytes = ctypes.c_size_t(0)
            _check(_lib().qx_gemv_fused_workspace(ctypes.byref(nbytes)), "qx_gemv_fused_workspace")
            self._ws = torch.zeros(int(nbytes.value) + 256, dtype=torch.uint8, device=dev)
            off = (-self._ws.data_ptr()) % 256
            self._ws_args = (ctypes.c_void_p(self._ws.data_ptr() + off), int(nbytes.value))

    def __call__(self):
        if self._ws is not None:
            _check(_lib().qx_gemv_fused(*self._args, *self._ws_args, _stream(self._dev)), "qx_gemv_fused")
        else:
            _check(_lib().qx_gemv_chain(*self._args, _stream(self._dev)), "qx_gemv_chain")


class DecodeStep(GemvChain):
    """A whole decode step as one qx_decode_step call (qx_decode_step_fused
    with `fused`): the host-to-device
    copies `h2d` [(device tensor, host tensor)], the groups of a GemvChain, the
    device-to-host copies `d2h` [(host tensor, device tensor)], then (sync) a
    synchronization of the stream.  Host tensors should be pinned.  Arguments
    are bound once; build a new step if a tensor is replaced."""

    def __init__(self, groups, h2d=(), d2h=(), pdl: bool = True, sync: bool = True, fused: bool = False,
                 separate: bool = False):
        super().__init__(groups, pdl, fused, separate)

        def copies(pairs, to_device):
            arr = []
            for dst, src in pairs:
                if _on_device(dst) != to_device or _on_device(src) == to_device:
                    raise ValueError("h2d pairs are (device, host), d2h pairs (host, device)")
                if not (dst.is_contiguous() and src.is_contiguous()):
                    raise ValueError("copies need contiguous tensors")
                nb = src.numel() * src.element_size()
                if dst.numel() * dst.element_size() != nb:
                    raise ValueError("a copy's two tensors differ in size")
                arr.append(_Copy(dst.data_ptr(), src.data_ptr(), nb))
                self._keep += [dst, src]
            return ((_Copy * len(arr))(*arr) if arr else None), len(arr)

        self._in, nin = copies(list(h2d), True)
        self._out, nout = copies(list(d2h), False)
        groups_arr, ng, batch, ydt, flags = self._args
        self._step = (self._in, nin, groups_arr, ng, batch, ydt, flags, self._out, nout, 1 if sync else 0)

    def __call__(self):
        if self._ws is not None:
            st = self._step
            _check(_lib().qx_decode_step_fused(*st[:7], *self._ws_args, *st[7:], _stream(self._dev)),
                   "qx_decode_step_fused")
        else:
            _check(_lib().qx_decode_step(*self._step, _stream(self._dev)), "qx_decode_step")


def gemm(P: PackedMatrix, X: torch.Tensor, out: torch.Tensor | None = None) -> torch.Tensor:
    """Prefill Y = X W_hat^T for X [m][k] (qx_gemm); returns fp16 [m][n]."""
    _dev_tensor(X, "X")
    m = X.shape[0]
    Y = out if out is not None else torch.empty((m, P.n), dtype=torch.float16, device=X.device)
    _dev_tensor(Y, "out")
    pc = P.c()
    _check(_lib().qx_gemm(ctypes.byref(pc), _ptr(X), m, _ptr(Y), _stream(X.device)), "qx_gemm")
    return Y


def gemm_splitk_workspace_bytes(n: int, k: int, m: int, recipe: Recipe) -> int:
    """Workspace bytes qx_gemm_splitk needs on the current device (0: no split)."""
    b = ctypes.c_size_t(0)
    r = recipe.c()
    _check(_lib().qx_gemm_splitk_workspace(n, k, m, ctypes.byref(r), ctypes.byref(b)), "qx_gemm_splitk_workspace")
    return int(b.value)


def gemm_splitk_plan(n: int, k: int, m: int, num_sms: int) -> tuple:
    """(tokens per tile, k splits, workspace bytes) of qx_gemm_splitk (host only)."""
    bn, sp, nb = ctypes.c_int32(0), ctypes.c_int32(0), ctypes.c_size_t(0)
    _check(_lib().qx_gemm_splitk_plan(n, k, m, num_sms, ctypes.byref(bn), ctypes.byref(sp), ctypes.byref(nb)),
           "qx_gemm_splitk_plan")
    return bn.value, sp.value, int(nb.value)


_WORKSPACES: dict = {}


def splitk_workspace(device, nbytes: int) -> torch.Tensor:
    """A zero-filled workspace of at least `nbytes` for `device`, kept per
    device and current stream (calls on one stream run one after another, so
    they may share it; qx_gemm_splitk leaves it zero-filled)."""
    dev = torch.device(device)
    key = (dev.index, torch.cuda.current_stream(dev).cuda_stream)
    ws = _WORKSPACES.get(key)
    if ws is None or ws.numel() < nbytes:
        ws = torch.zeros(max(nbytes, 256), dtype=torch.uint8, device=dev)
        _WORKSPACES[key] = ws
    return ws


def gemm_splitk(P: PackedMatrix, X: torch.Tensor, out: torch.Tensor | None = None,
                workspace: torch.Tensor | None = None, pdl: bool = False) -> torch.Tensor:
    """Y = X W_hat^T with k split across CTAs when the tiles alone leave SMs
    idle (qx_gemm_splitk): the tensor-core decode path for 1..16 rows of X and
    the path for short prefills.  ``pdl`` lets the kernel start while the
    previous kernel in the stream runs: set it only when that kernel does not
    write these weights.  Returns fp16 [m][n]."""
    _dev_tensor(X, "X")
    m = X.shape[0]
    Y = out if out is not None else torch.empty((m, P.n), dtype=torch.float16, device=X.device)
    _dev_tensor(Y, "out")
    need = gemm_splitk_workspace_bytes(P.n, P.k, m, P.recipe)
    ws = workspace if workspace is not None else splitk_workspace(X.device, need)
    if not _on_device(ws) or ws.dtype != torch.uint8:
        raise ValueError("workspace must be a CUDA uint8 tensor")
    pc = P.c()
    _check(_lib().qx_gemm_splitk(ctypes.byref(pc), _ptr(X), m, _ptr(Y), _ptr(ws), ws.numel(),
                                 GEMM_PDL if pdl else 0, _stream(X.device)), "qx_gemm_splitk")
    return Y


def gemm_splitk_noalloc(P: PackedMatrix, X: torch.Tensor, out: torch.Tensor | None = None) -> torch.Tensor:
    """qx_gemm_splitk without a workspace (qx_gemm_splitk_noalloc): the library's
    static 4 MiB scratch holds the partial tiles.  Returns fp16 [m][n]."""
    _dev_tensor(X, "X")
    m = X.shape[0]
    Y = out if out is not None else torch.empty((m, P.n), dtype=torch.float16, device=X.device)
    _dev_tensor(Y, "out")
    pc = P.c()
    _check(_lib().qx_gemm_splitk_noalloc(ctypes.byref(pc), _ptr(X), m, _ptr(Y), _stream(X.device)),
           "qx_gemm_splitk_noalloc")
    return Y


def quantize_act(x: torch.Tensor):
    """Per-token int8 activations (qx_quantize_act): returns (q int8 [b][k], scales fp32 [b])."""
    _dev_tensor(x, "x")
    x2 = x.view(-1, x.shape[-1])
    b, k = x2.shape
    q = torch.empty((b, k), dtype=torch.int8, device=x.device)
    s = torch.empty((b,), dtype=torch.float32, device=x.device)
    _check(_lib().qx_quantize_act(_ptr(x2), b, k, _ptr(q), _ptr(s), _stream(x.device)), "qx_quantize_act")
    return q, s


def dequant_act(q: torch.Tensor, scales: torch.Tensor, out: torch.Tensor | None = None) -> torch.Tensor:
    """fp16 x_hat = fp16(fp32(s_b q)) [m][k] of int8 activations (qx_dequant_act)."""
    if not _on_device(q) or q.dtype != torch.int8 or not q.is_contiguous():
        raise ValueError("q must be a contiguous CUDA int8 tensor")
    _dev_tensor(scales, "scales", torch.float32)
    m, k = q.shape
    xh = out if out is not None else torch.empty((m, k), dtype=torch.float16, device=q.device)
    _dev_tensor(xh, "out")
    _check(_lib().qx_dequant_act(_ptr(q), _ptr(scales), m, k, _ptr(xh), _stream(q.device)), "qx_dequant_act")
    return xh


def gemm_a8(P, x: torch.Tensor, out: torch.Tensor | None = None, splitk: bool = False) -> torch.Tensor:
    """W.A8 prefill Y = x_hat W_hat^T: per-token int8 activations
    (qx_quantize_act), their fp16 form (qx_dequant_act), then the tensor-core
    matmul (qx_gemm, qx_gemm_splitk with ``splitk``, or qx_q4x_gemm for a
    Q4xMatrix).  Returns fp16 [m][n]."""
    q, s = quantize_act(x)
    xh = dequant_act(q, s)
    if isinstance(P, Q4xMatrix):
        return q4x_gemm_splitk(P, xh, out=out) if splitk else q4x_gemm(P, xh, out=out)
    return gemm_splitk(P, xh, out=out) if splitk else gemm(P, xh, out=out)


def gemv_a8(P: PackedMatrix, q: torch.Tensor, scales: torch.Tensor, out: torch.Tensor | None = None,
            out_dtype=torch.float16) -> torch.Tensor:
    """W.A8 decode y = s_b x (q_w - z) q x s_g (qx_gemv_a8) for uniform weights; returns [batch][n]."""
    if not _on_device(q) or q.dtype != torch.int8 or not q.is_contiguous():
        raise ValueError("q must be a contiguous CUDA int8 tensor")
    _dev_tensor(scales, "scales", torch.float32)
    b = q.shape[0]
    dt = out.dtype if out is not None else out_dtype
    y = out if out is not None else torch.empty((b, P.n), dtype=dt, device=q.device)
    _dev_tensor(y, "out", dt)
    pc = P.c()
    _check(_lib().qx_gemv_a8(ctypes.byref(pc), _ptr(q), _ptr(scales), b, _ptr(y), F32 if dt == torch.float32 else F16,
                             _stream(q.device)), "qx_gemv_a8")
    return y


def select_recipe(W: torch.Tensor, candidates, max_bpw: float | None = None):
    """Per-matrix recipe choice by the exact Frobenius error (qx_select_recipe).

    Returns ``(index or None, errors, bpws)``: errors[i] is sum (w - w_hat)^2 in
    units of 2^-48 as an exact int (None over the budget)."""
    _dev_tensor(W, "W")
    n, k = W.shape
    cands = list(candidates)
    arr = (_Recipe * len(cands))(*[r.c() for r in cands])
    nbytes = ctypes.c_size_t(0)
    _check(_lib().qx_select_workspace(n, k, arr, len(cands), ctypes.byref(nbytes)), "qx_select_workspace")
    ws = torch.empty(max(int(nbytes.value), 256), dtype=torch.uint8, device=W.device)
    chosen = ctypes.c_int32(-1)
    err = (ctypes.c_uint64 * (2 * len(cands)))()
    bpw = (ctypes.c_double * len(cands))()
    _check(_lib().qx_select_recipe(_ptr(W), n, k, arr, len(cands), float(max_bpw or 0.0), _ptr(ws), ws.numel(),
                                   ctypes.byref(chosen), err, bpw, _stream(W.device)), "qx_select_recipe")
    errors = [None if err[2 * i] == err[2 * i + 1] == 2 ** 64 - 1 else err[2 * i] | (err[2 * i + 1] << 64)
              for i in range(len(cands))]
    return (None if chosen.value < 0 else chosen.value), errors, list(bpw)


Q4X_GROUP = 64


def q4x_size(n: int, k: int) -> dict:
    """Byte sizes of the Q4X buffers of an n x k matrix (host-only call)."""
    s = _Q4xSizes()
    _check(_lib().qx_q4x_size(n, k, ctypes.byref(s)), "qx_q4x_size")
    return {"codes": s.codes, "scales": s.scales, "books": s.books, "codebooks": s.codebooks}


def q4x_workspace_bytes(n: int, k: int) -> int:
    nbytes = ctypes.c_size_t(0)
    _check(_lib().qx_q4x_workspace(n, k, ctypes.byref(nbytes)), "qx_q4x_workspace")
    return int(nbytes.value)


class Q4xMatrix:
    """A Q4X shared-codebook matrix (4-bit codes, fp16 scale and 2-bit book
    index per group of 64, four 16-level codebooks), in torch device tensors."""

    def __init__(self, n, k, codes, scales, books, codebooks):
        self.n, self.k = int(n), int(k)
        self.codes, self.scales, self.books, self.codebooks = codes, scales, books, codebooks

    @classmethod
    def empty(cls, n: int, k: int, device) -> "Q4xMatrix":
        sz = q4x_size(n, k)
        return cls(n, k, torch.empty(sz["codes"], dtype=torch.uint8, device=device),
                   torch.empty(sz["scales"] // 2, dtype=torch.float16, device=device),
                   torch.empty(sz["books"], dtype=torch.uint8, device=device),
                   torch.empty(sz["codebooks"] // 2, dtype=torch.float16, device=device))

    @property
    def device(self):
        return self.codes.device

    def nbytes(self) -> int:
        return sum(t.numel() * t.element_size() for t in (self.codes, self.scales, self.books, self.codebooks))

    def c(self) -> _Q4x:
        return _Q4x(self.n, self.k, *(t.data_ptr() for t in (self.codes, self.scales, self.books, self.codebooks)))

    def to_numpy(self) -> dict:
        """Host copies in the oracle's array shapes (for tests)."""
        G = self.k // Q4X_GROUP
        return {"codes": self.codes.cpu().numpy().reshape(self.n, -1),
                "scales": self.scales.cpu().numpy().reshape(self.n, G),
                "books": self.books.cpu().numpy().reshape(self.n, -1),
                "codebooks": self.codebooks.cpu().numpy().reshape(4, 16)}


def q4x_quantize(W: torch.Tensor, iters: int = 25, out: Q4xMatrix | None = None) -> Q4xMatrix:
    """Learn the four codebooks of fp16 W [n][k] and code it (qx_q4x_quantize)."""
    _dev_tensor(W, "W")
    n, k = W.shape
    P = out if out is not None else Q4xMatrix.empty(n, k, W.device)
    ws = torch.empty(q4x_workspace_bytes(n, k), dtype=torch.uint8, device=W.device)
    pc = P.c()
    _check(_lib().qx_q4x_quantize(_ptr(W), iters, ctypes.byref(pc), _ptr(ws), ws.numel(), _stream(W.device)),
           "qx_q4x_quantize")
    return P


def q4x_dequant(P: Q4xMatrix, out: torch.Tensor | None = None) -> torch.Tensor:
    """fp16 W_hat [n][k] of a Q4X matrix (qx_q4x_dequant)."""
    W = out if out is not None else torch.empty((P.n, P.k), dtype=torch.float16, device=P.device)
    _dev_tensor(W, "out")
    pc = P.c()
    _check(_lib().qx_q4x_dequant(ctypes.byref(pc), _ptr(W), _stream(P.device)), "qx_q4x_dequant")
    return W


def q4x_gemv(P: Q4xMatrix, x: torch.Tensor, out: torch.Tensor | None = None,
             out_dtype=torch.float16) -> torch.Tensor:
    """Decode y = x W_hat^T for a Q4X matrix, x [batch][k] (qx_q4x_gemv)."""
    _dev_tensor(x, "x")
    x2 = x.view(-1, P.k)
    b = x2.shape[0]
    dt = out.dtype if out is not None else out_dtype
    y = out if out is not None else torch.empty((b, P.n), dtype=dt, device=x.device)
    _dev_tensor(y, "out", dt)
    pc = P.c()
    _check(_lib().qx_q4x_gemv(ctypes.byref(pc), _ptr(x2), b, _ptr(y), F32 if dt == torch.float32 else F16,
                              _stream(x.device)), "qx_q4x_gemv")
    return y


def q4x_gemv_multi(mats, xs, outs=None, out_dtype=torch.float16):
    """Several Q4X decode matmuls in one launch (qx_q4x_gemv_multi): y[i] =
    xs[i] W_hat_i^T for up to eight matrices; returns the outputs."""
    mats, xs = list(mats), list(xs)
    if len(mats) != len(xs) or not 1 <= len(mats) <= 8:
        raise ValueError("1..8 matrices, one x per matrix")
    x2 = [x.view(-1, P.k) for P, x in zip(mats, xs)]
    for x in x2:
        _dev_tensor(x, "x")
    b = x2[0].shape[0]
    if any(x.shape[0] != b for x in x2):
        raise ValueError("every x must have the same batch")
    dt = outs[0].dtype if outs is not None else out_dtype
    ys = list(outs) if outs is not None else [torch.empty((b, P.n), dtype=dt, device=x2[0].device) for P in mats]
    for y in ys:
        _dev_tensor(y, "out", dt)
    cnt = len(mats)
    arr = (_Q4x * cnt)(*[P.c() for P in mats])
    xa = (ctypes.c_void_p * cnt)(*[x.data_ptr() for x in x2])
    ya = (ctypes.c_void_p * cnt)(*[y.data_ptr() for y in ys])
    _check(_lib().qx_q4x_gemv_multi(arr, cnt, xa, b, ya, F32 if dt == torch.float32 else F16,
                                    _stream(x2[0].device)), "qx_q4x_gemv_multi")
    return ys


def selftest_wait_timeout(limit_us: int, device=None) -> None:
    """Launch the failure-detection self-test (qx_selftest_wait_timeout): a
    bounded wait that runs out; device_status() then returns 5 (QX_ERR_TIMEOUT)."""
    dev = device if device is not None else torch.device("cuda", torch.cuda.current_device())
    _check(_lib().qx_selftest_wait_timeout(int(limit_us), _stream(dev)), "qx_selftest_wait_timeout")


def q4x_gemm(P: Q4xMatrix, X: torch.Tensor, out: torch.Tensor | None = None) -> torch.Tensor:
    """Prefill Y = X W_hat^T for a Q4X matrix on the tensor cores (qx_q4x_gemm); fp16 [m][n]."""
    _dev_tensor(X, "X")
    m = X.shape[0]
    Y = out if out is not None else torch.empty((m, P.n), dtype=torch.float16, device=X.device)
    _dev_tensor(Y, "out")
    pc = P.c()
    _check(_lib().qx_q4x_gemm(ctypes.byref(pc), _ptr(X), m, _ptr(Y), _stream(X.device)), "qx_q4x_gemm")
    return Y


def q4x_gemm_splitk(P: Q4xMatrix, X: torch.Tensor, out: torch.Tensor | None = None,
                    workspace: torch.Tensor | None = None, pdl: bool = False) -> torch.Tensor:
    """qx_q4x_gemm with k split across CTAs when the tiles leave SMs idle
    (qx_q4x_gemm_splitk); the workspace is kept per device and stream as for
    gemm_splitk.  Returns fp16 [m][n]."""
    _dev_tensor(X, "X")
    m = X.shape[0]
    Y = out if out is not None else torch.empty((m, P.n), dtype=torch.float16, device=X.device)
    _dev_tensor(Y, "out")
    need = ctypes.c_size_t(0)
    _check(_lib().qx_q4x_gemm_splitk_workspace(P.n, P.k, m, ctypes.byref(need)), "qx_q4x_gemm_splitk_workspace")
    ws = workspace if workspace is not None else splitk_workspace(X.device, int(need.value))
    pc = P.c()
    _check(_lib().qx_q4x_gemm_splitk(ctypes.byref(pc), _ptr(X), m, _ptr(Y), _ptr(ws), ws.numel(),
                                     GEMM_PDL if pdl else 0, _stream(X.device)), "qx_q4x_gemm_splitk")
    return Y


def recipe_table(path: str) -> dict:
    """A per-matrix recipe table (JSON, as recipes/llava_v1_6_7b.json): for
    each sub-model, its layer count and a list of (name, n, k, Recipe); the
    recipe is chosen per matrix (Sections 2.1, 2.3)."""
    import json

    kinds = {"uniform": UNIFORM, "lut": LUT}
    with open(path) as f:
        t = json.load(f)
    out = {}
    for sub, body in t.items():
        if not isinstance(body, dict) or "matrices" not in body:
            continue
        mats = [(m["name"], int(m["n"]), int(m["k"]),
                 Recipe(int(m["recipe"]["bits"]), int(m["recipe"]["group_size"]), kinds[m["recipe"]["kind"]]))
                for m in body["matrices"]]
        out[sub] = {"layers": int(body["layers"]), "matrices": mats}
    return out


# ------------------------------------------------------------ save / load
# A packed matrix on disk: an 80-byte little-endian header, then its four
# buffers in header order.
#   magic "QXPK", u16 version (1), u16 format (0: per-group codes, 1: Q4X),
#   i64 n, i64 k, i32 bits, group_size, kind, lloyd_iters,
#   u64 sizes of the four buffers (codes, scales, zeros | books, luts | codebooks),
#   u32 CRC-32 of the buffers in order, u32 zero.
_HDR = "<4sHHqqiiiiQQQQII"
_MAGIC, _VERSION = b"QXPK", 1


def _bytes_of(t):
    return b"" if t is None else t.detach().contiguous().cpu().view(torch.uint8).numpy().tobytes()


def save(path: str, P) -> None:
    """Write a PackedMatrix or Q4xMatrix (its buffers copied to the host)."""
    import struct
    import zlib

    if isinstance(P, Q4xMatrix):
        fmt, rec = 1, (4, Q4X_GROUP, 0, 0)
        bufs = [P.codes, P.scales, P.books, P.codebooks]
    elif isinstance(P, PackedMatrix):
        fmt, rec = 0, (P.recipe.bits, P.recipe.group_size, P.recipe.kind, P.recipe.lloyd_iters)
        bufs = [P.codes, P.scales, P.zeros, P.luts]
    else:
        raise TypeError("save takes a PackedMatrix or a Q4xMatrix")
    raw = [_bytes_of(t) for t in bufs]
    crc = 0
    for r in raw:
        crc = zlib.crc32(r, crc)
    hdr = struct.pack(_HDR, _MAGIC, _VERSION, fmt, P.n, P.k, *rec, *[len(r) for r in raw], crc, 0)
    with open(path, "wb") as f:
        f.write(hdr)
        for r in raw:
            f.write(r)


def load(path: str, device=None):
    """Read a matrix written by :func:`save` onto `device` (a torch device;
    default the current CUDA device).  Raises ValueError on a bad magic,
    version or checksum, or sizes that disagree with the library's layout."""
    import struct
    import zlib

    with open(path, "rb") as f:
        blob = f.read()
    size = struct.calcsize(_HDR)
    if len(blob) < size:
        raise ValueError("truncated header")
    magic, ver, fmt, n, k, bits, g, kind, iters, s0, s1, s2, s3, crc, _ = struct.unpack_from(_HDR, blob)
    if magic != _MAGIC or ver != _VERSION or fmt not in (0, 1):
        raise ValueError("not a qx packed matrix (magic, version or format)")
    sizes = [s0, s1, s2, s3]
    if fmt == 1:
        want = q4x_size(n, k)
        expect = [want["codes"], want["scales"], want["books"], want["codebooks"]]
    else:
        rec = Recipe(bits, g, kind, iters)
        want = packed_size(n, k, rec)
        expect = [want["codes"], want["scales"], want["zeros"], want["luts"]]
    if sizes != expect:
        raise ValueError("buffer sizes disagree with the layout of this shape and recipe")
    if len(blob) != size + sum(sizes):
        raise ValueError("file length disagrees with the header")
    c, off, raw = 0, size, []
    for sz in sizes:
        raw.append(blob[off:off + sz])
        c = zlib.crc32(raw[-1], c)
        off += sz
    if c != crc:
        raise ValueError("checksum mismatch")
    dev = device if device is not None else torch.device("cuda", torch.cuda.current_device())

    def tensor(r, dtype):
        if not r:
            return None
        return torch.frombuffer(bytearray(r), dtype=torch.uint8).view(dtype).to(dev)

    if fmt == 1:
        return Q4xMatrix(n, k, tensor(raw[0], torch.uint8), tensor(raw[1], torch.float16),
                         tensor(raw[2], torch.uint8), tensor(raw[3], torch.float16))
    return PackedMatrix(n, k, rec, tensor(raw[0], torch.uint8), tensor(raw[1], torch.float16),
                        tensor(raw[2], torch.uint8), tensor(raw[3], torch.float16))


def device_status(stream=None) -> int:
    """Synchronize and return/clear the device status (0 = QX_OK)."""
    s = ctypes.c_void_p(stream.cuda_stream) if stream is not None else _stream(torch.device("cuda"))
    return _lib().qx_get_device_status(s)


def version() -> int:
    return _lib().qx_version()
