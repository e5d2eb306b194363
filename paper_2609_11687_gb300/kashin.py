"""Python binding of libkashin (include/kashin.h).

Argument marshalling only: device memory comes from PyTorch tensors, streams
from ``torch.cuda``; every step of the decomposition, coding, transform and
reconstruction runs in the library's CUDA kernels.  Importing this module loads
``libkashin.so`` from this package directory and raises ``ImportError`` if it is
missing -- there is no fallback implementation.

Two layers:

* ``kd_*`` functions mirror the C entry points one to one (raw device pointers
  as Python ints, a status code back);
* tensor-level wrappers take and return torch tensors: ``decompose`` (and
  ``decompose_batch``, ``decompose_batch_host``), ``apply_p`` (``apply_p_batch``,
  ``prepare_p`` + ``apply_p_prepared``), ``reconstruct`` (``reconstruct_batch``),
  ``dequantise`` (``dequantise_batch``), ``rht``, and the products from the 2-bit
  planes ``matmul_2bit`` (fp32) and ``matmul_2bit_f16`` (fp16 or bf16 activations,
  tensor cores), each with a ``_batch`` form.
"""

from __future__ import annotations

import ctypes
import dataclasses
import os
from typing import Optional

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libkashin.so")

KD_OK, KD_ERR_INVALID_ARG, KD_ERR_UNSUPPORTED_N, KD_ERR_CUDA, KD_ERR_NONFINITE, KD_ERR_WORKSPACE, KD_ERR_TIMEOUT = range(7)
KD_F32, KD_F16, KD_BF16 = 0, 1, 2
KD_VEC_ROWS, KD_VEC_COLUMNS = 0, 1

EXPORTS = ("kd_status_string", "kd_version", "kd_supported", "kd_tuned", "kd_workspace_size", "kd_signs",
           "kd_decompose", "kd_apply_p", "kd_reconstruct", "kd_read_status", "kd_decompose_static",
           "kd_read_status_static", "kd_staging_size_host", "kd_decompose_batch_host",
           "kd_matmul_2bit", "kd_matmul_2bit_batch", "kd_matmul_2bit_f16", "kd_matmul_2bit_f16_batch",
           "kd_matmul_2bit_bf16", "kd_matmul_2bit_bf16_batch",
           "kd_apply_p_batch", "kd_prepare_p", "kd_apply_p_prepared",
           "kd_rht_block", "kd_rht", "kd_dequantise", "kd_dequantise_batch", "kd_measure_fp32_peak",
           "kd_workspace_size_batch", "kd_decompose_batch", "kd_reconstruct_batch")
KD_MAX_BATCH = 32


class KdPlane(ctypes.Structure):
    """kd_plane: one 2-bit code plane to expand (kd_dequantise_batch)."""
    _fields_ = [("codes", ctypes.c_void_p), ("centres", ctypes.c_void_p), ("out", ctypes.c_void_p),
                ("m", ctypes.c_int64), ("ld", ctypes.c_int64)]


class KdRecMat(ctypes.Structure):
    """kd_recmat: one matrix to re-materialise (kd_reconstruct_batch)."""
    _fields_ = [("codes_u", ctypes.c_void_p), ("codes_v", ctypes.c_void_p), ("centres_u", ctypes.c_void_p),
                ("centres_v", ctypes.c_void_p), ("sign_seed", ctypes.c_uint64), ("w_hat", ctypes.c_void_p),
                ("m", ctypes.c_int64), ("ld", ctypes.c_int64)]


class KdPMat(ctypes.Structure):
    """Mirror of kd_pmat (include/kashin.h): rows x -> y = P x with one sign seed."""
    _fields_ = [("x", ctypes.c_void_p), ("y", ctypes.c_void_p), ("m", ctypes.c_int64), ("sign_seed", ctypes.c_uint64)]


class KdFoldMat(ctypes.Structure):
    """Mirror of kd_fold_mat (include/kashin.h): one matrix of kd_matmul_2bit_batch."""
    _fields_ = [("codes_u", ctypes.c_void_p), ("codes_v", ctypes.c_void_p), ("centres_u", ctypes.c_void_p),
                ("centres_v", ctypes.c_void_p), ("x", ctypes.c_void_p), ("xp", ctypes.c_void_p),
                ("y", ctypes.c_void_p), ("n", ctypes.c_int64), ("m", ctypes.c_int64), ("ldx", ctypes.c_int64),
                ("ldy", ctypes.c_int64)]


class KdFoldMatF16(ctypes.Structure):
    """Mirror of kd_fold_mat_f16 (include/kashin.h): one matrix of kd_matmul_2bit_f16_batch."""
    _fields_ = KdFoldMat._fields_


class KdMatrixHost(ctypes.Structure):
    """Mirror of kd_matrix_host (include/kashin.h): every pointer is host memory."""
    _fields_ = [("w", ctypes.c_void_p), ("m", ctypes.c_int64), ("ld", ctypes.c_int64),
                ("sign_seed", ctypes.c_uint64), ("codes_u", ctypes.c_void_p), ("codes_v", ctypes.c_void_p),
                ("centres_u", ctypes.c_void_p), ("centres_v", ctypes.c_void_p), ("coeffs", ctypes.c_void_p)]


class KdMatrix(ctypes.Structure):
    """Mirror of kd_matrix (include/kashin.h)."""
    _fields_ = [("w", ctypes.c_void_p), ("m", ctypes.c_int64), ("ld", ctypes.c_int64),
                ("sign_seed", ctypes.c_uint64), ("codes_u", ctypes.c_void_p), ("codes_v", ctypes.c_void_p),
                ("centres_u", ctypes.c_void_p), ("centres_v", ctypes.c_void_p), ("coeffs", ctypes.c_void_p)]


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built; run paper_2609_11687_gb300.build.build() "
                          "(the CUDA library is required, there is no CPU fallback)")
    lib = ctypes.CDLL(LIB_PATH)
    c_i64, c_u64, c_int, c_vp, c_sz = ctypes.c_int64, ctypes.c_uint64, ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t
    lib.kd_status_string.argtypes = [c_int]
    lib.kd_status_string.restype = ctypes.c_char_p
    lib.kd_version.argtypes = []
    lib.kd_version.restype = ctypes.c_char_p
    lib.kd_supported.argtypes = [c_i64]
    lib.kd_supported.restype = c_int
    lib.kd_tuned.argtypes = [c_i64]
    lib.kd_tuned.restype = c_int
    lib.kd_workspace_size.argtypes = [c_i64]
    lib.kd_workspace_size.restype = c_sz
    lib.kd_signs.argtypes = [c_u64, c_i64, c_vp]
    lib.kd_signs.restype = c_int
    lib.kd_decompose.argtypes = [c_vp, c_int, c_int, c_i64, c_i64, c_i64, c_u64, c_int, c_int,
                                 c_vp, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp, c_sz, c_vp]
    lib.kd_decompose.restype = c_int
    lib.kd_apply_p.argtypes = [c_vp, c_vp, c_i64, c_i64, c_u64, c_vp, c_sz, c_vp]
    lib.kd_apply_p.restype = c_int
    lib.kd_reconstruct.argtypes = [c_vp, c_vp, c_vp, c_vp, c_i64, c_i64, c_u64, c_int, c_int, c_vp,
                                   c_i64, c_vp, c_sz, c_vp]
    lib.kd_reconstruct.restype = c_int
    lib.kd_read_status.argtypes = [c_vp, c_vp]
    lib.kd_read_status.restype = c_int
    lib.kd_decompose_static.argtypes = [c_vp, c_int, c_int, c_i64, c_i64, c_i64, c_u64, c_int, c_int,
                                        c_vp, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp]
    lib.kd_decompose_static.restype = c_int
    lib.kd_read_status_static.argtypes = [c_vp]
    lib.kd_read_status_static.restype = c_int
    lib.kd_staging_size_host.argtypes = [c_vp, c_int, c_int, c_int, c_i64]
    lib.kd_staging_size_host.restype = c_sz
    lib.kd_decompose_batch_host.argtypes = [c_vp, c_int, c_int, c_int, c_i64, c_int, c_int, c_vp, c_sz, c_vp,
                                            c_sz, c_vp]
    lib.kd_decompose_batch_host.restype = c_int
    lib.kd_matmul_2bit.argtypes = [c_vp, c_vp, c_vp, c_vp, c_i64, c_i64, c_vp, c_vp, c_i64, c_i64, c_vp, c_i64, c_vp]
    lib.kd_matmul_2bit.restype = c_int
    lib.kd_matmul_2bit_batch.argtypes = [c_vp, c_int, c_i64, c_vp]
    lib.kd_matmul_2bit_batch.restype = c_int
    lib.kd_prepare_p.argtypes = [c_vp, c_int, c_i64, c_vp, ctypes.c_size_t, c_vp]
    lib.kd_prepare_p.restype = c_int
    lib.kd_apply_p_prepared.argtypes = [c_vp, c_int, c_i64, c_vp, ctypes.c_size_t, c_vp]
    lib.kd_apply_p_prepared.restype = c_int
    lib.kd_matmul_2bit_f16.argtypes = [c_vp, c_vp, c_vp, c_vp, c_i64, c_i64, c_vp, c_vp, c_i64, c_i64, c_vp, c_i64,
                                       c_vp]
    lib.kd_matmul_2bit_f16.restype = c_int
    lib.kd_matmul_2bit_f16_batch.argtypes = [c_vp, c_int, c_i64, c_vp]
    lib.kd_matmul_2bit_f16_batch.restype = c_int
    lib.kd_matmul_2bit_bf16.argtypes = lib.kd_matmul_2bit_f16.argtypes
    lib.kd_matmul_2bit_bf16.restype = c_int
    lib.kd_matmul_2bit_bf16_batch.argtypes = [c_vp, c_int, c_i64, c_vp]
    lib.kd_matmul_2bit_bf16_batch.restype = c_int
    lib.kd_apply_p_batch.argtypes = [c_vp, c_int, c_i64, c_vp, c_sz, c_vp]
    lib.kd_apply_p_batch.restype = c_int
    lib.kd_workspace_size_batch.argtypes = [c_i64, c_int]
    lib.kd_workspace_size_batch.restype = c_sz
    lib.kd_decompose_batch.argtypes = [c_vp, c_int, c_int, c_int, c_i64, c_int, c_int, c_vp, c_sz, c_vp]
    lib.kd_decompose_batch.restype = c_int
    lib.kd_reconstruct_batch.argtypes = [c_vp, c_int, c_i64, c_int, c_int, c_vp, c_sz, c_vp]
    lib.kd_reconstruct_batch.restype = c_int
    lib.kd_measure_fp32_peak.argtypes = [c_vp, c_vp]
    lib.kd_measure_fp32_peak.restype = c_int
    lib.kd_dequantise.argtypes = [c_vp, c_vp, c_i64, c_i64, c_int, c_int, c_vp, c_i64, c_vp]
    lib.kd_dequantise.restype = c_int
    lib.kd_dequantise_batch.argtypes = [c_vp, c_int, c_i64, c_int, c_int, c_vp]
    lib.kd_dequantise_batch.restype = c_int
    lib.kd_rht_block.argtypes = [c_i64]
    lib.kd_rht_block.restype = c_i64
    lib.kd_rht.argtypes = [c_vp, c_int, c_i64, c_i64, c_i64, c_u64, c_int, c_vp, c_i64, c_vp, c_vp]
    lib.kd_rht.restype = c_int
    return lib


lib = _load()


class KashinError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)}")


def status_string(s: int) -> str:
    return lib.kd_status_string(int(s)).decode()


def version() -> str:
    return lib.kd_version().decode()


# ---------------------------------------------------------------------------
# one-to-one mirrors of the C entry points
# ---------------------------------------------------------------------------

def kd_supported(n: int) -> int:
    return lib.kd_supported(int(n))


def kd_tuned(n: int) -> bool:
    return bool(lib.kd_tuned(int(n)))


def kd_workspace_size(n: int) -> int:
    return int(lib.kd_workspace_size(int(n)))


def kd_signs(sign_seed: int, n: int) -> np.ndarray:
    out = np.empty(int(n), dtype=np.int8)
    st = lib.kd_signs(ctypes.c_uint64(int(sign_seed) & ((1 << 64) - 1)), int(n), out.ctypes.data)
    if st != KD_OK:
        raise KashinError(st, "kd_signs")
    return out


def kd_decompose(w, dtype, layout, n, m, ld, sign_seed, iters, kmeans_iters, codes_u, codes_v, centres_u,
                 centres_v, coeffs, u, vhat, resid, trace, workspace, ws_bytes, stream) -> int:
    return lib.kd_decompose(w, dtype, layout, n, m, ld, ctypes.c_uint64(int(sign_seed) & ((1 << 64) - 1)),
                            iters, kmeans_iters, codes_u, codes_v, centres_u, centres_v, coeffs, u, vhat, resid,
                            trace, workspace, ws_bytes, stream)


def kd_apply_p(x, y, n, m, sign_seed, workspace, ws_bytes, stream) -> int:
    return lib.kd_apply_p(x, y, n, m, ctypes.c_uint64(int(sign_seed) & ((1 << 64) - 1)), workspace, ws_bytes,
                          stream)


def kd_reconstruct(codes_u, codes_v, centres_u, centres_v, n, m, sign_seed, out_dtype, layout, w_hat, ld,
                   workspace, ws_bytes, stream) -> int:
    return lib.kd_reconstruct(codes_u, codes_v, centres_u, centres_v, n, m,
                              ctypes.c_uint64(int(sign_seed) & ((1 << 64) - 1)), out_dtype, layout, w_hat, ld,
                              workspace, ws_bytes, stream)


def kd_batchable(n: int) -> bool:
    """True when kd_decompose_batch runs all matrices of length n in one launch
    (tuned lengths n <= 8192, as include/kashin.h states); longer vectors and the
    run-time-length path run one launch each."""
    return kd_tuned(n) and int(n) <= 8192


def kd_workspace_size_batch(n: int, count: int) -> int:
    return int(lib.kd_workspace_size_batch(int(n), int(count)))


def kd_decompose_batch(mats, count, dtype, layout, n, iters, kmeans_iters, workspace, ws_bytes, stream) -> int:
    return lib.kd_decompose_batch(mats, count, dtype, layout, n, iters, kmeans_iters, workspace, ws_bytes, stream)


def kd_reconstruct_batch(mats, count, n, out_dtype, layout, workspace, ws_bytes, stream) -> int:
    return lib.kd_reconstruct_batch(mats, count, n, out_dtype, layout, workspace, ws_bytes, stream)


def kd_read_status(workspace, stream) -> int:
    return lib.kd_read_status(workspace, stream)


def kd_decompose_static(w, dtype, layout, n, m, ld, sign_seed, iters, kmeans_iters, codes_u, codes_v, centres_u,
                        centres_v, coeffs, u, vhat, resid, trace, stream) -> int:
    return lib.kd_decompose_static(w, dtype, layout, n, m, ld, ctypes.c_uint64(int(sign_seed) & ((1 << 64) - 1)),
                                   iters, kmeans_iters, codes_u, codes_v, centres_u, centres_v, coeffs, u, vhat,
                                   resid, trace, stream)


def kd_read_status_static(stream) -> int:
    return lib.kd_read_status_static(stream)


def kd_staging_size_host(mats, count, dtype, layout, n) -> int:
    return int(lib.kd_staging_size_host(mats, count, dtype, layout, n))


def kd_decompose_batch_host(mats, count, dtype, layout, n, iters, kmeans_iters, staging, staging_bytes, workspace,
                            ws_bytes, stream) -> int:
    return lib.kd_decompose_batch_host(mats, count, dtype, layout, n, iters, kmeans_iters, staging, staging_bytes,
                                       workspace, ws_bytes, stream)


def kd_dequantise(codes, centres, n, m, out_dtype, layout, out, ld, stream) -> int:
    return lib.kd_dequantise(codes, centres, n, m, out_dtype, layout, out, ld, stream)


def kd_dequantise_batch(planes, count, n, out_dtype, layout, stream) -> int:
    return lib.kd_dequantise_batch(planes, count, n, out_dtype, layout, stream)


def measure_fp32_peak(stream=None) -> float:
    """Measured FP32 TFLOP/s of the current device (packed FFMA chains)."""
    out = ctypes.c_double(0.0)
    st = lib.kd_measure_fp32_peak(ctypes.byref(out), _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_measure_fp32_peak")
    return out.value


def kd_rht_block(n) -> int:
    return int(lib.kd_rht_block(int(n)))


def kd_rht(x, dtype, n, m, ldx, seed, inverse, y, ldy, status, stream) -> int:
    return lib.kd_rht(x, dtype, n, m, ldx, ctypes.c_uint64(int(seed) & ((1 << 64) - 1)), inverse, y, ldy, status,
                      stream)


# ---------------------------------------------------------------------------
# torch-tensor wrappers
# ---------------------------------------------------------------------------

def _torch():
    import torch
    return torch


def _dtype_code(t) -> int:
    torch = _torch()
    m = {torch.float32: KD_F32, torch.float16: KD_F16, torch.bfloat16: KD_BF16}
    if t not in m:
        raise TypeError(f"unsupported dtype {t}")
    return m[t]


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _ld(t) -> int:
    """Row stride of a 2-D tensor for the C ABI: a single row's stride is never used, so
    report its length (torch and numpy may give a one-row tensor any row stride)."""
    return t.stride(0) if t.shape[0] > 1 else t.shape[1]


def _stream(stream) -> int:
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


class Workspace:
    """Device scratch for one vector length (reusable across calls on one stream)."""

    def __init__(self, n: int, device="cuda", count: int = 1):
        torch = _torch()
        self.n = int(n)
        self.count = int(count)
        size = kd_workspace_size(self.n) if self.count == 1 else kd_workspace_size_batch(self.n, self.count)
        if size == 0:
            raise KashinError(KD_ERR_UNSUPPORTED_N if kd_supported(self.n) else KD_ERR_CUDA,
                              f"kd_workspace_size({self.n})")
        self.nbytes = size
        self.buf = torch.empty(size, dtype=torch.uint8, device=device)

    @property
    def ptr(self) -> int:
        return self.buf.data_ptr()


@dataclasses.dataclass
class Decomposed:
    codes_u: "object"     # int32 view of uint32 words, (m, ceil(n/16))
    codes_v: "object"
    centres_u: "object"   # float32 (m, 4)
    centres_v: "object"
    coeffs: "object"      # float32 (m, 4) or None
    u: "object"           # float32 (m, n) or None
    vhat: "object"
    resid: "object"
    trace: "object"       # int8 (m, 4*iters + 2*kmeans_iters, n) or None


def decompose(w, iters: int, sign_seed: int, layout: str = "rows", factors: bool = False,
              coeffs: bool = True, trace: bool = False, workspace: Optional[Workspace] = None,
              out: Optional[Decomposed] = None, stream=None, kmeans_iters: int = 0) -> Decomposed:
    """Decompose every vector of ``w`` (Alg. 1) and 2-bit code both factors
    (closed-form centres, then ``kmeans_iters`` Lloyd refinement iterations).

    ``layout='rows'``: ``w`` is (m, n), vector j = ``w[j]`` (nn.Linear weight).
    ``layout='columns'``: ``w`` is (n, m), vector j = ``w[:, j]`` (the paper's W).
    """
    torch = _torch()
    if not w.is_cuda:
        raise ValueError("w must be a CUDA tensor")
    if w.dim() != 2 or w.stride(1) != 1:
        raise ValueError("w must be 2-D with unit inner stride")
    lay = KD_VEC_ROWS if layout == "rows" else KD_VEC_COLUMNS
    if lay == KD_VEC_ROWS:
        m, n = w.shape
    else:
        n, m = w.shape
    ld = _ld(w)
    dev = w.device
    words = (n + 15) // 16
    if out is None:
        f32 = dict(dtype=torch.float32, device=dev)
        out = Decomposed(
            codes_u=torch.empty((m, words), dtype=torch.int32, device=dev),
            codes_v=torch.empty((m, words), dtype=torch.int32, device=dev),
            centres_u=torch.empty((m, 4), **f32), centres_v=torch.empty((m, 4), **f32),
            coeffs=torch.empty((m, 4), **f32) if coeffs else None,
            u=torch.empty((m, n), **f32) if factors else None,
            vhat=torch.empty((m, n), **f32) if factors else None,
            resid=torch.empty((m, n), **f32) if factors else None,
            trace=torch.empty((m, 4 * iters + 2 * kmeans_iters, n), dtype=torch.int8, device=dev) if trace else None)
    ws = workspace if workspace is not None else Workspace(n, dev)
    st = kd_decompose(w.data_ptr(), _dtype_code(w.dtype), lay, n, m, ld, sign_seed, int(iters), int(kmeans_iters),
                      _ptr(out.codes_u), _ptr(out.codes_v), _ptr(out.centres_u), _ptr(out.centres_v),
                      _ptr(out.coeffs), _ptr(out.u), _ptr(out.vhat), _ptr(out.resid), _ptr(out.trace),
                      ws.ptr, ws.nbytes, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_decompose")
    return out


def decompose_batch(ws, iters: int, sign_seeds, layout: str = "rows", coeffs: bool = False,
                    workspace: Optional[Workspace] = None, outs=None, stream=None, kmeans_iters: int = 0):
    """Decompose and code several matrices of one vector length in one launch
    (kd_decompose_batch): ``ws`` is a list of up to KD_MAX_BATCH CUDA tensors of one
    dtype and layout, ``sign_seeds`` their seeds.  Returns one Decomposed per matrix
    (no factor or trace outputs)."""
    torch = _torch()
    if not 1 <= len(ws) <= KD_MAX_BATCH or len(sign_seeds) != len(ws):
        raise ValueError(f"1..{KD_MAX_BATCH} matrices with one seed each")
    lay = KD_VEC_ROWS if layout == "rows" else KD_VEC_COLUMNS
    n = ws[0].shape[1] if lay == KD_VEC_ROWS else ws[0].shape[0]
    dt = ws[0].dtype
    arr = (KdMatrix * len(ws))()
    res = []
    for i, w in enumerate(ws):
        if not w.is_cuda or w.dim() != 2 or w.stride(1) != 1 or w.dtype != dt:
            raise ValueError("matrices must be 2-D CUDA tensors of one dtype with unit inner stride")
        m = w.shape[0] if lay == KD_VEC_ROWS else w.shape[1]
        if (w.shape[1] if lay == KD_VEC_ROWS else w.shape[0]) != n:
            raise ValueError("matrices must share the vector length")
        if outs is not None:
            o = outs[i]
        else:
            f32 = dict(dtype=torch.float32, device=w.device)
            o = Decomposed(codes_u=torch.empty((m, (n + 15) // 16), dtype=torch.int32, device=w.device),
                           codes_v=torch.empty((m, (n + 15) // 16), dtype=torch.int32, device=w.device),
                           centres_u=torch.empty((m, 4), **f32), centres_v=torch.empty((m, 4), **f32),
                           coeffs=torch.empty((m, 4), **f32) if coeffs else None,
                           u=None, vhat=None, resid=None, trace=None)
        arr[i] = KdMatrix(w.data_ptr(), m, _ld(w), int(sign_seeds[i]) & ((1 << 64) - 1),
                          _ptr(o.codes_u), _ptr(o.codes_v), _ptr(o.centres_u), _ptr(o.centres_v), _ptr(o.coeffs))
        res.append(o)
    wsp = workspace if workspace is not None else Workspace(n, ws[0].device, count=len(ws))
    st = kd_decompose_batch(ctypes.cast(arr, ctypes.c_void_p), len(ws), _dtype_code(dt), lay, n, int(iters),
                            int(kmeans_iters), wsp.ptr, wsp.nbytes, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_decompose_batch")
    return res


def kd_matmul_2bit(codes_u, codes_v, centres_u, centres_v, n, m, x, xp, batch, ldx, y, ldy, stream) -> int:
    return lib.kd_matmul_2bit(codes_u, codes_v, centres_u, centres_v, n, m, x, xp, batch, ldx, y, ldy, stream)


def matmul_2bit(dec: "Decomposed", x, xp, out=None, stream=None):
    """``Y = X W_hat^T`` from the code planes (App. C): ``x`` and ``xp`` (= apply_p of the
    rows of x with the matrix's sign seed) are fp32 CUDA tensors (batch, n); returns
    (batch, m) fp32."""
    torch = _torch()
    m, words = dec.codes_u.shape
    if x.dim() != 2 or x.dtype != torch.float32 or xp.shape != x.shape or xp.dtype != x.dtype:
        raise ValueError("x and xp must be fp32 (batch, n) tensors of one shape")
    if x.stride(1) != 1 or xp.stride(1) != 1 or _ld(x) != _ld(xp):
        raise ValueError("x and xp need unit inner stride and equal row strides")
    b, n = x.shape
    if (n + 15) // 16 != words:
        raise ValueError("x does not match the code planes' vector length")
    y = out if out is not None else torch.empty((b, m), dtype=torch.float32, device=x.device)
    st = kd_matmul_2bit(dec.codes_u.data_ptr(), dec.codes_v.data_ptr(), dec.centres_u.data_ptr(),
                        dec.centres_v.data_ptr(), n, m, x.data_ptr(), xp.data_ptr(), b, _ld(x), y.data_ptr(),
                        _ld(y), _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_matmul_2bit")
    return y


def kd_matmul_2bit_batch(mats, count, batch, stream) -> int:
    return lib.kd_matmul_2bit_batch(mats, count, batch, stream)


def kd_matmul_2bit_f16(codes_u, codes_v, centres_u, centres_v, n, m, x, xp, batch, ldx, y, ldy, stream) -> int:
    return lib.kd_matmul_2bit_f16(codes_u, codes_v, centres_u, centres_v, n, m, x, xp, batch, ldx, y, ldy, stream)


def kd_matmul_2bit_f16_batch(mats, count, batch, stream) -> int:
    return lib.kd_matmul_2bit_f16_batch(mats, count, batch, stream)


def kd_matmul_2bit_bf16(codes_u, codes_v, centres_u, centres_v, n, m, x, xp, batch, ldx, y, ldy, stream) -> int:
    return lib.kd_matmul_2bit_bf16(codes_u, codes_v, centres_u, centres_v, n, m, x, xp, batch, ldx, y, ldy, stream)


def kd_matmul_2bit_bf16_batch(mats, count, batch, stream) -> int:
    return lib.kd_matmul_2bit_bf16_batch(mats, count, batch, stream)


def matmul_2bit_f16(dec: "Decomposed", x, xp, out=None, stream=None):
    """kd_matmul_2bit_f16 (or _bf16): ``Y = X W_hat^T`` from the code planes on the tensor
    cores, for fp16 (or bf16) ``x`` and ``xp`` (batch, n) CUDA tensors; returns (batch, m) fp32."""
    return matmul_2bit_f16_batch([dec], [x], [xp], outs=None if out is None else [out], stream=stream)[0]


def matmul_2bit_f16_batch(decs, xs, xps, outs=None, stream=None):
    """kd_matmul_2bit_f16_batch (or _bf16_batch, for bf16 inputs): ``Y_i = X_i W_hat_i^T``
    for several matrices, 16-bit inputs of one type and batch size, one launch per 16 rows."""
    torch = _torch()
    dt = xs[0].dtype
    if dt not in (torch.float16, torch.bfloat16):
        raise ValueError("x must be fp16 or bf16")
    if not 1 <= len(decs) <= KD_MAX_BATCH or len(xs) != len(decs) or len(xps) != len(decs):
        raise ValueError(f"1..{KD_MAX_BATCH} matrices with one x and one xp each")
    b = xs[0].shape[0]
    arr = (KdFoldMatF16 * len(decs))()
    res = []
    for i, (d, x, xp) in enumerate(zip(decs, xs, xps)):
        m, words = d.codes_u.shape
        if x.dim() != 2 or x.shape[0] != b or x.dtype != dt or xp.shape != x.shape \
                or xp.dtype != x.dtype or x.stride(1) != 1 or xp.stride(1) != 1 or _ld(x) != _ld(xp):
            raise ValueError("x and xp must be 16-bit (batch, n) tensors of one type and shape, unit inner stride")
        n = x.shape[1]
        if (n + 15) // 16 != words:
            raise ValueError("x does not match the code planes' vector length")
        y = outs[i] if outs is not None else torch.empty((b, m), dtype=torch.float32, device=x.device)
        arr[i] = KdFoldMatF16(d.codes_u.data_ptr(), d.codes_v.data_ptr(), d.centres_u.data_ptr(),
                              d.centres_v.data_ptr(), x.data_ptr(), xp.data_ptr(), y.data_ptr(), n, m, _ld(x),
                              _ld(y))
        res.append(y)
    call = kd_matmul_2bit_bf16_batch if dt == torch.bfloat16 else kd_matmul_2bit_f16_batch
    st = call(ctypes.cast(arr, ctypes.c_void_p), len(decs), b, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_matmul_2bit_bf16_batch" if dt == torch.bfloat16 else "kd_matmul_2bit_f16_batch")
    return res


def kd_apply_p_batch(mats, count, n, workspace, ws_bytes, stream) -> int:
    return lib.kd_apply_p_batch(mats, count, n, workspace, ws_bytes, stream)


def matmul_2bit_batch(decs, xs, xps, outs=None, stream=None):
    """kd_matmul_2bit_batch: ``Y_i = X_i W_hat_i^T`` for several matrices in one launch
    (``decs`` Decomposed, ``xs``/``xps`` fp32 (batch, n_i) CUDA tensors, one batch size)."""
    torch = _torch()
    if not 1 <= len(decs) <= KD_MAX_BATCH or len(xs) != len(decs) or len(xps) != len(decs):
        raise ValueError(f"1..{KD_MAX_BATCH} matrices with one x and one xp each")
    b = xs[0].shape[0]
    arr = (KdFoldMat * len(decs))()
    res = []
    for i, (d, x, xp) in enumerate(zip(decs, xs, xps)):
        m, words = d.codes_u.shape
        if x.dim() != 2 or x.shape[0] != b or x.dtype != torch.float32 or xp.shape != x.shape \
                or xp.dtype != x.dtype or x.stride(1) != 1 or xp.stride(1) != 1 or _ld(x) != _ld(xp):
            raise ValueError("x and xp must be fp32 (batch, n) tensors of one shape, unit inner stride")
        n = x.shape[1]
        if (n + 15) // 16 != words:
            raise ValueError("x does not match the code planes' vector length")
        y = outs[i] if outs is not None else torch.empty((b, m), dtype=torch.float32, device=x.device)
        arr[i] = KdFoldMat(d.codes_u.data_ptr(), d.codes_v.data_ptr(), d.centres_u.data_ptr(), d.centres_v.data_ptr(),
                           x.data_ptr(), xp.data_ptr(), y.data_ptr(), n, m, _ld(x), _ld(y))
        res.append(y)
    st = kd_matmul_2bit_batch(ctypes.cast(arr, ctypes.c_void_p), len(decs), b, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_matmul_2bit_batch")
    return res


def apply_p_batch(xs, sign_seeds, outs=None, workspace: Optional[Workspace] = None, stream=None):
    """kd_apply_p_batch: ``y = P x`` for the rows of several fp32 (m_i, n) tensors, each
    with its own sign seed, in one launch."""
    torch = _torch()
    if not 1 <= len(xs) <= KD_MAX_BATCH or len(sign_seeds) != len(xs):
        raise ValueError(f"1..{KD_MAX_BATCH} matrices with one seed each")
    n = xs[0].shape[1]
    arr = (KdPMat * len(xs))()
    res = []
    for i, x in enumerate(xs):
        if x.dtype != torch.float32 or not x.is_contiguous() or x.dim() != 2 or x.shape[1] != n:
            raise ValueError("inputs must be contiguous fp32 (m, n) CUDA tensors of one n")
        y = outs[i] if outs is not None else torch.empty_like(x)
        arr[i] = KdPMat(x.data_ptr(), y.data_ptr(), x.shape[0], int(sign_seeds[i]) & ((1 << 64) - 1))
        res.append(y)
    ws = workspace if workspace is not None else Workspace(n, xs[0].device, count=len(xs))
    st = kd_apply_p_batch(ctypes.cast(arr, ctypes.c_void_p), len(xs), n, ws.ptr, ws.nbytes, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_apply_p_batch")
    return res


def kd_prepare_p(seeds, count, n, workspace, ws_bytes, stream) -> int:
    return lib.kd_prepare_p(seeds, count, n, workspace, ws_bytes, stream)


def kd_apply_p_prepared(mats, count, n, workspace, ws_bytes, stream) -> int:
    return lib.kd_apply_p_prepared(mats, count, n, workspace, ws_bytes, stream)


def prepare_p(n: int, sign_seeds, workspace: Optional[Workspace] = None, device="cuda", stream=None) -> Workspace:
    """kd_prepare_p: P's twiddle table and the sign sets of ``sign_seeds`` written once
    into a workspace (returned) for apply_p_prepared."""
    if not 1 <= len(sign_seeds) <= KD_MAX_BATCH:
        raise ValueError(f"1..{KD_MAX_BATCH} sign seeds")
    ws = workspace if workspace is not None else Workspace(n, device, count=len(sign_seeds))
    seeds = (ctypes.c_uint64 * len(sign_seeds))(*[int(s) & ((1 << 64) - 1) for s in sign_seeds])
    st = kd_prepare_p(ctypes.cast(seeds, ctypes.c_void_p), len(sign_seeds), n, ws.ptr, ws.nbytes, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_prepare_p")
    return ws


def apply_p_prepared(xs, workspace: Workspace, outs=None, stream=None):
    """kd_apply_p_prepared: ``y_i = P_i x_i`` with the tables prepare_p left in
    ``workspace`` (matrix i takes sign set i)."""
    torch = _torch()
    if not 1 <= len(xs) <= KD_MAX_BATCH:
        raise ValueError(f"1..{KD_MAX_BATCH} matrices")
    n = xs[0].shape[1]
    arr = (KdPMat * len(xs))()
    res = []
    for i, x in enumerate(xs):
        if x.dtype != torch.float32 or not x.is_contiguous() or x.dim() != 2 or x.shape[1] != n:
            raise ValueError("inputs must be contiguous fp32 (m, n) CUDA tensors of one n")
        y = outs[i] if outs is not None else torch.empty_like(x)
        arr[i] = KdPMat(x.data_ptr(), y.data_ptr(), x.shape[0], 0)
        res.append(y)
    st = kd_apply_p_prepared(ctypes.cast(arr, ctypes.c_void_p), len(xs), n, workspace.ptr, workspace.nbytes,
                             _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_apply_p_prepared")
    return res


def _host_descriptors(ws, sign_seeds, layout, outs):
    """kd_matrix_host array for host tensors ``ws`` and host outputs ``outs`` (one
    Decomposed of CPU tensors per matrix)."""
    if not 1 <= len(ws) <= KD_MAX_BATCH or len(sign_seeds) != len(ws) or len(outs) != len(ws):
        raise ValueError(f"1..{KD_MAX_BATCH} matrices with one seed and one output set each")
    lay = KD_VEC_ROWS if layout == "rows" else KD_VEC_COLUMNS
    n = ws[0].shape[1] if lay == KD_VEC_ROWS else ws[0].shape[0]
    arr = (KdMatrixHost * len(ws))()
    for i, (w, o) in enumerate(zip(ws, outs)):
        if w.is_cuda or w.dim() != 2 or w.stride(1) != 1 or w.dtype != ws[0].dtype:
            raise ValueError("matrices must be 2-D host tensors of one dtype with unit inner stride")
        m = w.shape[0] if lay == KD_VEC_ROWS else w.shape[1]
        for t in (o.codes_u, o.codes_v, o.centres_u, o.centres_v, o.coeffs):
            if t is not None and t.is_cuda:
                raise ValueError("outputs must be host tensors")
        arr[i] = KdMatrixHost(w.data_ptr(), m, _ld(w), int(sign_seeds[i]) & ((1 << 64) - 1),
                              _ptr(o.codes_u), _ptr(o.codes_v), _ptr(o.centres_u), _ptr(o.centres_v),
                              _ptr(o.coeffs))
    return arr, lay, n


def host_outputs(m: int, n: int, coeffs: bool = False, pin: bool = True) -> Decomposed:
    """Host (pinned) output tensors for one matrix of decompose_batch_host."""
    torch = _torch()
    def mk(shape, dt):
        t = torch.empty(shape, dtype=dt)
        return t.pin_memory() if pin else t
    return Decomposed(codes_u=mk((m, (n + 15) // 16), torch.int32), codes_v=mk((m, (n + 15) // 16), torch.int32),
                      centres_u=mk((m, 4), torch.float32), centres_v=mk((m, 4), torch.float32),
                      coeffs=mk((m, 4), torch.float32) if coeffs else None, u=None, vhat=None, resid=None,
                      trace=None)


def staging_size_host(ws, layout: str = "rows", coeffs: bool = False) -> int:
    """Device staging bytes decompose_batch_host needs for host matrices ``ws``."""
    lay = KD_VEC_ROWS if layout == "rows" else KD_VEC_COLUMNS
    n = ws[0].shape[1] if lay == KD_VEC_ROWS else ws[0].shape[0]
    outs = [host_outputs(w.shape[0] if lay == KD_VEC_ROWS else w.shape[1], n, coeffs, pin=False) for w in ws]
    arr, lay, n = _host_descriptors(ws, [0] * len(ws), layout, outs)
    return kd_staging_size_host(ctypes.cast(arr, ctypes.c_void_p), len(ws), _dtype_code(ws[0].dtype), lay, n)


def decompose_batch_host(ws, iters: int, sign_seeds, outs, staging, workspace: Workspace, layout: str = "rows",
                         stream=None, kmeans_iters: int = 0):
    """kd_decompose_batch_host: host matrices ``ws`` (pinned CPU tensors) in, host
    outputs ``outs`` (from host_outputs) written once ``stream`` completes.  ``staging``
    is a device uint8 tensor of at least staging_size_host(ws) bytes."""
    arr, lay, n = _host_descriptors(ws, sign_seeds, layout, outs)
    st = kd_decompose_batch_host(ctypes.cast(arr, ctypes.c_void_p), len(ws), _dtype_code(ws[0].dtype), lay, n,
                                 int(iters), int(kmeans_iters), staging.data_ptr(),
                                 staging.numel() * staging.element_size(), workspace.ptr, workspace.nbytes,
                                 _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_decompose_batch_host")
    return outs


def read_status(workspace: Workspace, stream=None) -> int:
    return kd_read_status(workspace.ptr, _stream(stream))


def apply_p(x, sign_seed: int, out=None, workspace: Optional[Workspace] = None, stream=None):
    """``y_j = P x_j`` for the rows of the fp32 (m, n) tensor ``x``."""
    torch = _torch()
    if x.dtype != torch.float32 or not x.is_contiguous() or x.dim() != 2:
        raise ValueError("x must be a contiguous fp32 (m, n) CUDA tensor")
    m, n = x.shape
    y = out if out is not None else torch.empty_like(x)
    ws = workspace if workspace is not None else Workspace(n, x.device)
    st = kd_apply_p(x.data_ptr(), y.data_ptr(), n, m, sign_seed, ws.ptr, ws.nbytes, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_apply_p")
    return y


def dequantise(codes, centres, n: int, dtype=None, layout: str = "rows", out=None, stream=None):
    """Dense factor matrix from one 2-bit code plane and its centres (App. C):
    (m, n) for layout "rows", (n, m) for "columns"."""
    torch = _torch()
    dtype = dtype or torch.float32
    m = codes.shape[0]
    lay = KD_VEC_ROWS if layout == "rows" else KD_VEC_COLUMNS
    if out is None:
        out = torch.empty((m, n) if lay == KD_VEC_ROWS else (n, m), dtype=dtype, device=codes.device)
    st = kd_dequantise(codes.data_ptr(), centres.data_ptr(), n, m, _dtype_code(out.dtype), lay, out.data_ptr(),
                       _ld(out), _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_dequantise")
    return out


def dequantise_batch(planes, n: int, dtype=None, layout: str = "rows", outs=None, stream=None):
    """``dequantise`` for several (codes, centres) planes of one vector length in one
    launch (kd_dequantise_batch); returns one dense matrix per plane."""
    torch = _torch()
    if not 1 <= len(planes) <= KD_MAX_BATCH:
        raise ValueError(f"1..{KD_MAX_BATCH} planes")
    dtype = dtype or torch.float32
    lay = KD_VEC_ROWS if layout == "rows" else KD_VEC_COLUMNS
    arr = (KdPlane * len(planes))()
    res = []
    for i, (codes, centres) in enumerate(planes):
        m = codes.shape[0]
        if outs is not None:
            o = outs[i]
        else:
            o = torch.empty((m, n) if lay == KD_VEC_ROWS else (n, m), dtype=dtype, device=codes.device)
        if o.dtype != dtype:
            raise ValueError("outputs must share one dtype")
        arr[i] = KdPlane(codes.data_ptr(), centres.data_ptr(), o.data_ptr(), m, _ld(o))
        res.append(o)
    st = kd_dequantise_batch(ctypes.cast(arr, ctypes.c_void_p), len(planes), n, _dtype_code(dtype), lay,
                             _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_dequantise_batch")
    return res


def rht(x, seed: int, inverse: bool = False, out=None, status=None, stream=None):
    """Randomized-Hadamard rotation of the rows of the (m, n) tensor ``x`` (fp32,
    fp16 or bf16, unit inner stride) into an fp32 (m, n) tensor; ``out=x`` rotates
    an fp32 tensor in place (Sec. 4, Kashin-DCT+H).  ``status``: optional int32
    device tensor of one element that collects KD_RHT_ERR_* bits."""
    torch = _torch()
    if x.dim() != 2 or x.stride(1) != 1:
        raise ValueError("x must be a 2-D CUDA tensor with unit inner stride")
    m, n = x.shape
    y = out if out is not None else torch.empty((m, n), dtype=torch.float32, device=x.device)
    if y.dtype != torch.float32 or y.shape != x.shape or y.stride(1) != 1:
        raise ValueError("out must be an fp32 tensor of x's shape with unit inner stride")
    st = kd_rht(x.data_ptr(), _dtype_code(x.dtype), n, m, _ld(x), seed, 1 if inverse else 0, y.data_ptr(),
                _ld(y), status.data_ptr() if status is not None else None, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_rht")
    return y


def reconstruct(dec: Decomposed, n: int, sign_seed: int, dtype=None, layout: str = "rows", out=None,
                workspace: Optional[Workspace] = None, stream=None):
    """Dense ``W_hat = U_q + P V_q`` from codes and centres (App. C)."""
    torch = _torch()
    dtype = dtype or torch.float32
    m = dec.codes_u.shape[0]
    lay = KD_VEC_ROWS if layout == "rows" else KD_VEC_COLUMNS
    dev = dec.codes_u.device
    if out is None:
        out = torch.empty((m, n) if lay == KD_VEC_ROWS else (n, m), dtype=dtype, device=dev)
    ws = workspace if workspace is not None else Workspace(n, dev)
    st = kd_reconstruct(dec.codes_u.data_ptr(), dec.codes_v.data_ptr(), dec.centres_u.data_ptr(),
                        dec.centres_v.data_ptr(), n, m, sign_seed, _dtype_code(out.dtype), lay, out.data_ptr(),
                        _ld(out), ws.ptr, ws.nbytes, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_reconstruct")
    return out


def reconstruct_batch(decs, n: int, sign_seeds, dtype=None, layout: str = "rows", outs=None,
                      workspace: Optional[Workspace] = None, stream=None):
    """``reconstruct`` for several decomposed matrices of one vector length in one
    launch (kd_reconstruct_batch); returns one dense W_hat per matrix."""
    torch = _torch()
    if not 1 <= len(decs) <= KD_MAX_BATCH or len(sign_seeds) != len(decs):
        raise ValueError(f"1..{KD_MAX_BATCH} matrices with one seed each")
    dtype = dtype or torch.float32
    lay = KD_VEC_ROWS if layout == "rows" else KD_VEC_COLUMNS
    dev = decs[0].codes_u.device
    arr = (KdRecMat * len(decs))()
    res = []
    for i, d in enumerate(decs):
        m = d.codes_u.shape[0]
        o = outs[i] if outs is not None else torch.empty((m, n) if lay == KD_VEC_ROWS else (n, m), dtype=dtype,
                                                         device=dev)
        if o.dtype != dtype:
            raise ValueError("outputs must share one dtype")
        arr[i] = KdRecMat(d.codes_u.data_ptr(), d.codes_v.data_ptr(), d.centres_u.data_ptr(), d.centres_v.data_ptr(),
                          int(sign_seeds[i]) & ((1 << 64) - 1), o.data_ptr(), m, _ld(o))
        res.append(o)
    ws = workspace if workspace is not None else Workspace(n, dev, count=len(decs))
    st = kd_reconstruct_batch(ctypes.cast(arr, ctypes.c_void_p), len(decs), n, _dtype_code(dtype), lay, ws.ptr,
                              ws.nbytes, _stream(stream))
    if st != KD_OK:
        raise KashinError(st, "kd_reconstruct_batch")
    return res


def unpack_codes(words, n: int):
    """(m, ceil(n/16)) int32 words -> (m, n) int64 codes (host numpy)."""
    w = np.asarray(words.cpu().numpy() if hasattr(words, "cpu") else words).astype(np.uint32).astype(np.uint64)
    m = w.shape[0]
    idx = np.arange(n)
    return ((w[:, idx // 16] >> (2 * (idx % 16)).astype(np.uint64)) & np.uint64(3)).astype(np.int64).reshape(m, n)
