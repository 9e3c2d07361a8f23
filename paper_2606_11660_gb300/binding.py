"""Thin ctypes binding of the C ABI in include/bergson.h.

Each ``bergson_*`` function here has the name of the C entry point it calls
and only marshals arguments: torch tensors become device pointers and leading
dimensions, ``stream=None`` becomes torch's current stream.  All computation
happens in the CUDA library; if the library is missing, loading it raises.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
from typing import Optional, Sequence

_PKG_DIR = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG_DIR, "libbergson.so")

BERGSON_OK = 0
BERGSON_EINVAL = -1
BERGSON_EALIGN = -2
BERGSON_EUNSUPPORTED = -3
BERGSON_EWORKSPACE = -4
BERGSON_ECUDA = -5
BERGSON_EDEVICE_TIMEOUT = -6
BERGSON_EMOMENT = -7

BERGSON_PROJ_GAUSSIAN = 0
BERGSON_PROJ_IDENTITY = 1
BERGSON_PROJ_RADEMACHER = 2
BERGSON_PROJ_UNIFORM = 3

BERGSON_LAYER_BIAS = 1

BERGSON_AGG_SUM = 0
BERGSON_AGG_MEAN = 1

BERGSON_FISHER_INV_SQRT = 0
BERGSON_FISHER_INV = 1

STATUS_NAMES = {
    0: "BERGSON_OK", -1: "BERGSON_EINVAL", -2: "BERGSON_EALIGN", -3: "BERGSON_EUNSUPPORTED",
    -4: "BERGSON_EWORKSPACE", -5: "BERGSON_ECUDA", -6: "BERGSON_EDEVICE_TIMEOUT",
    -7: "BERGSON_EMOMENT",
}

# Every symbol include/bergson.h declares.
EXPORTED = (
    "bergson_project_grads_workspace", "bergson_project_grads", "bergson_build_store",
    "bergson_score_topk_workspace", "bergson_score_topk", "bergson_score_bottomk",
    "bergson_projection_matrix",
    "bergson_module_seeds", "bergson_sync_status", "bergson_last_error", "bergson_version",
    "bergson_debug_wait_probe", "bergson_debug_inject_status", "bergson_debug_project_plan",
    "bergson_debug_score_plan", "bergson_debug_xgemm_plan", "bergson_project_grads_noalloc",
    "bergson_score_grads_workspace", "bergson_score_grads", "bergson_token_scores_workspace",
    "bergson_token_scores", "bergson_aggregate_rows_workspace", "bergson_aggregate_rows",
    "bergson_fisher_fit_workspace", "bergson_fisher_fit", "bergson_fisher_preconditioner_workspace",
    "bergson_fisher_preconditioner", "bergson_precondition_rows", "bergson_store_save",
    "bergson_store_load", "bergson_fisher_preconditioner_tol", "bergson_debug_attr_once",
    "bergson_build_store_blocks", "bergson_score_topk_update_workspace",
    "bergson_score_topk_update", "bergson_score_bottomk_update",
    "bergson_score_topk_host_workspace", "bergson_score_topk_host",
)


class BergsonError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class bergson_layer(ctypes.Structure):
    _fields_ = [
        ("A", ctypes.c_void_p), ("G", ctypes.c_void_p),
        ("d_in", ctypes.c_int64), ("d_out", ctypes.c_int64),
        ("k_in", ctypes.c_int64), ("k_out", ctypes.c_int64),
        ("seed_in", ctypes.c_uint64), ("seed_out", ctypes.c_uint64),
        ("proj_kind", ctypes.c_int32), ("flags", ctypes.c_int32),
        ("r", ctypes.c_void_p), ("c", ctypes.c_void_p),
        ("out_col_offset", ctypes.c_int64), ("bias_col_offset", ctypes.c_int64),
    ]


_LIB = None


def lib() -> ctypes.CDLL:
    """The loaded library (raises if it was not built)."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
    L = ctypes.CDLL(LIB_PATH)
    i64, u64, vp, i32 = ctypes.c_int64, ctypes.c_uint64, ctypes.c_void_p, ctypes.c_int
    szp = ctypes.POINTER(ctypes.c_size_t)
    i64p = ctypes.POINTER(ctypes.c_int64)
    lp = ctypes.POINTER(bergson_layer)
    sig = {
        "bergson_project_grads_workspace": (i32, [lp, i32, i64, i64, szp]),
        "bergson_project_grads": (i32, [lp, i32, i64, i64, vp, vp, i64, vp, ctypes.c_size_t, vp]),
        "bergson_build_store": (i32, [vp, i64, i64, i64, i32, vp, i64, i64, i64, vp, vp]),
        "bergson_build_store_blocks": (i32, [vp, i64, i64, i64, i64p, i32, vp, i64, i64, i64,
                                             vp, vp]),
        "bergson_score_topk_workspace": (i32, [i64, i64, i64, i64, szp]),
        "bergson_score_topk": (i32, [vp, i64, i64, i64, vp, i64, i64, i64, vp, vp, vp,
                                     ctypes.c_size_t, vp]),
        "bergson_score_bottomk": (i32, [vp, i64, i64, i64, vp, i64, i64, i64, vp, vp, vp,
                                        ctypes.c_size_t, vp]),
        "bergson_score_topk_update_workspace": (i32, [i64, i64, i64, szp]),
        "bergson_score_topk_update": (i32, [vp, i64, i64, i64, i64, vp, i64, i64, i64, i32, vp,
                                            vp, vp, ctypes.c_size_t, vp]),
        "bergson_score_bottomk_update": (i32, [vp, i64, i64, i64, i64, vp, i64, i64, i64, i32,
                                               vp, vp, vp, ctypes.c_size_t, vp]),
        "bergson_score_topk_host_workspace": (i32, [i64, i64, i64, i64, szp]),
        "bergson_score_topk_host": (i32, [vp, i64, i64, i64, vp, i64, i64, i64, i32, i64, vp,
                                          vp, vp, ctypes.c_size_t, vp, vp]),
        "bergson_projection_matrix": (i32, [u64, i64, i64, i32, vp, vp, vp]),
        "bergson_module_seeds": (None, [u64, i64, ctypes.POINTER(u64), ctypes.POINTER(u64)]),
        "bergson_sync_status": (i32, [vp]),
        "bergson_last_error": (ctypes.c_char_p, []),
        "bergson_version": (i32, []),
        "bergson_debug_wait_probe": (i32, [u64, vp]),
        "bergson_debug_inject_status": (None, [i32, i32]),
        "bergson_debug_project_plan": (i32, [lp, i32, i64, i64, i64p, i64p, i64p, i64p]),
        "bergson_debug_score_plan": (i32, [i64, i64, i64, i64, i32, i64p, i32,
                                           ctypes.POINTER(i32)]),
        "bergson_debug_xgemm_plan": (i32, [i64, i64, i64, i64p, i32]),
        "bergson_debug_attr_once": (i32, [i32, i32, i32, i64p, ctypes.POINTER(i32)]),
        "bergson_project_grads_noalloc": (i32, [lp, i32, i64, i64, vp, vp, i64, vp]),
        "bergson_score_grads_workspace": (i32, [i64, i64, i64, szp]),
        "bergson_token_scores_workspace": (i32, [lp, i32, i64, i64, i64, szp]),
        "bergson_aggregate_rows_workspace": (i32, [i64, szp]),
        "bergson_store_save": (i32, [vp, i64, i64, i64, ctypes.c_char_p, i64, vp]),
        "bergson_store_load": (i32, [ctypes.c_char_p, i64, i64, i64, vp, i64, vp]),
        "bergson_fisher_fit_workspace": (i32, [i64, i64, szp]),
        "bergson_fisher_fit": (i32, [vp, i64, i64, i64, vp, i64, vp, ctypes.c_size_t, vp]),
        "bergson_fisher_preconditioner_workspace": (i32, [i64, szp]),
        "bergson_fisher_preconditioner": (i32, [vp, vp, i64, i64, ctypes.c_float, ctypes.c_float,
                                                i32, i32, vp, i64, vp, ctypes.c_size_t, vp]),
        "bergson_fisher_preconditioner_tol": (i32, [vp, vp, i64, i64, ctypes.c_float,
                                                    ctypes.c_float, i32, i32, ctypes.c_float, vp,
                                                    i64, vp, ctypes.c_size_t,
                                                    ctypes.POINTER(ctypes.c_float),
                                                    ctypes.POINTER(i32), vp]),
        "bergson_precondition_rows": (i32, [vp, i64, i64, i64, vp, i64, vp, i64, vp,
                                            ctypes.c_size_t, vp]),
        "bergson_aggregate_rows": (i32, [vp, i64, i64, i64, vp, i64, i32, i32, vp, i64, vp,
                                         ctypes.c_size_t, vp]),
        "bergson_token_scores": (i32, [lp, i32, i64, i64, vp, vp, i64, i64, vp, vp,
                                       ctypes.c_size_t, vp]),
        "bergson_score_grads": (i32, [vp, i64, i64, i64, vp, i64, i64, i32, vp, i64, vp,
                                      ctypes.c_size_t, vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _LIB = L
    return L


def bergson_last_error() -> str:
    return lib().bergson_last_error().decode()


def _check(status: int) -> None:
    if status != BERGSON_OK:
        raise BergsonError(status, bergson_last_error())


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    return t.data_ptr() if hasattr(t, "data_ptr") else int(t)


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


@dataclasses.dataclass
class Layer:
    """One nn.Linear's captured tensors: A [B,T,d_in] bf16, G [B,T,d_out] bf16."""
    A: object
    G: object
    k_in: int
    k_out: int
    seed_in: int
    seed_out: int
    r: object = None
    c: object = None
    out_col_offset: int = 0
    proj_kind: int = BERGSON_PROJ_GAUSSIAN
    bias_col_offset: Optional[int] = None     # set to also write the projected bias gradient

    def to_c(self) -> bergson_layer:
        bias = self.bias_col_offset is not None
        return bergson_layer(
            A=_ptr(self.A), G=_ptr(self.G), d_in=int(self.A.shape[-1]), d_out=int(self.G.shape[-1]),
            k_in=int(self.k_in), k_out=int(self.k_out), seed_in=int(self.seed_in),
            seed_out=int(self.seed_out), proj_kind=int(self.proj_kind),
            flags=BERGSON_LAYER_BIAS if bias else 0, r=_ptr(self.r), c=_ptr(self.c),
            out_col_offset=int(self.out_col_offset),
            bias_col_offset=int(self.bias_col_offset) if bias else 0)


def _layer_array(layers: Sequence) -> "ctypes.Array":
    arr = (bergson_layer * len(layers))()
    for i, ly in enumerate(layers):
        arr[i] = ly if isinstance(ly, bergson_layer) else ly.to_c()
    return arr


def bergson_module_seeds(base_seed: int, module_index: int) -> tuple[int, int]:
    a, b = ctypes.c_uint64(), ctypes.c_uint64()
    lib().bergson_module_seeds(int(base_seed), int(module_index), ctypes.byref(a), ctypes.byref(b))
    return a.value, b.value


def bergson_project_grads_workspace(layers: Sequence, B: int, T: int) -> int:
    arr = _layer_array(layers)
    n = ctypes.c_size_t()
    _check(lib().bergson_project_grads_workspace(arr, len(layers), int(B), int(T), ctypes.byref(n)))
    return n.value


def bergson_project_grads(layers: Sequence, B: int, T: int, mask, out, workspace,
                          stream=None, ld_out: Optional[int] = None) -> None:
    arr = _layer_array(layers)
    ld = int(out.stride(0)) if ld_out is None else int(ld_out)
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(lib().bergson_project_grads(arr, len(layers), int(B), int(T), _ptr(mask), _ptr(out), ld,
                                       _ptr(workspace), ws_bytes, _stream(stream)))


def bergson_project_grads_noalloc(layers: Sequence, B: int, T: int, mask, out, stream=None,
                                  ld_out: Optional[int] = None) -> None:
    """Like bergson_project_grads, but on the library's fixed static scratch (no workspace)."""
    arr = _layer_array(layers)
    ld = int(out.stride(0)) if ld_out is None else int(ld_out)
    _check(lib().bergson_project_grads_noalloc(arr, len(layers), int(B), int(T), _ptr(mask),
                                               _ptr(out), ld, _stream(stream)))


def bergson_build_store(proj, B: int, K: int, unit_normalize: bool, store, row_offset: int,
                        norms_out=None, stream=None) -> None:
    _check(lib().bergson_build_store(_ptr(proj), int(B), int(K), int(proj.stride(0)),
                                     1 if unit_normalize else 0, _ptr(store), int(store.stride(0)),
                                     int(row_offset), int(store.shape[0]), _ptr(norms_out),
                                     _stream(stream)))


def bergson_build_store_blocks(proj, B: int, K: int, block_offsets: Sequence[int], store,
                               row_offset: int, norms_out=None, stream=None) -> None:
    """Store rows with each column block [o_j, o_j+1) unit-normalised on its own."""
    n = len(block_offsets) - 1
    offs = (ctypes.c_int64 * max(1, n + 1))(*[int(v) for v in block_offsets])
    _check(lib().bergson_build_store_blocks(_ptr(proj), int(B), int(K), int(proj.stride(0)), offs,
                                            n, _ptr(store), int(store.stride(0)), int(row_offset),
                                            int(store.shape[0]), _ptr(norms_out), _stream(stream)))


def bergson_score_topk_workspace(N: int, K: int, Q: int, topk: int) -> int:
    n = ctypes.c_size_t()
    _check(lib().bergson_score_topk_workspace(int(N), int(K), int(Q), int(topk), ctypes.byref(n)))
    return n.value


def bergson_score_topk(store, N: int, K: int, queries, topk: int, out_scores, out_idx, workspace,
                       stream=None) -> None:
    Q = int(queries.shape[0])
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(lib().bergson_score_topk(_ptr(store), int(N), int(K), int(store.stride(0)),
                                    _ptr(queries), Q, int(queries.stride(0)), int(topk),
                                    _ptr(out_scores), _ptr(out_idx), _ptr(workspace), ws_bytes,
                                    _stream(stream)))


def bergson_score_bottomk(store, N: int, K: int, queries, bottomk: int, out_scores, out_idx,
                          workspace, stream=None) -> None:
    """The bottomk least similar store rows per query, lowest score first."""
    Q = int(queries.shape[0])
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(lib().bergson_score_bottomk(_ptr(store), int(N), int(K), int(store.stride(0)),
                                       _ptr(queries), Q, int(queries.stride(0)), int(bottomk),
                                       _ptr(out_scores), _ptr(out_idx), _ptr(workspace), ws_bytes,
                                       _stream(stream)))


def bergson_score_topk_update_workspace(K: int, Q: int, topk: int) -> int:
    n = ctypes.c_size_t()
    _check(lib().bergson_score_topk_update_workspace(int(K), int(Q), int(topk), ctypes.byref(n)))
    return n.value


def bergson_score_topk_update(store, N: int, K: int, row_base: int, queries, topk: int, init: bool,
                              scores, idx, workspace, stream=None, least: bool = False) -> None:
    """Merge the top-k (least: bottom-k) of store rows [row_base, row_base + N)
    (store[0:N] on the device) into the running result scores/idx [Q, topk]."""
    Q = int(queries.shape[0])
    fn = lib().bergson_score_bottomk_update if least else lib().bergson_score_topk_update
    _check(fn(_ptr(store), int(N), int(K), int(store.stride(0)), int(row_base), _ptr(queries), Q,
              int(queries.stride(0)), int(topk), 1 if init else 0, _ptr(scores), _ptr(idx),
              _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))


def bergson_score_topk_host_workspace(chunk_rows: int, K: int, Q: int, topk: int) -> int:
    n = ctypes.c_size_t()
    _check(lib().bergson_score_topk_host_workspace(int(chunk_rows), int(K), int(Q), int(topk),
                                                   ctypes.byref(n)))
    return n.value


def bergson_score_topk_host(host_store, N: int, K: int, queries, topk: int, chunk_rows: int,
                            out_scores, out_idx, workspace, stream=None, copy_stream=None,
                            least: bool = False) -> None:
    """Exact top-k (least: bottom-k) of a store in host memory (a CPU tensor,
    ideally pinned), streamed to the device in chunks of chunk_rows rows."""
    Q = int(queries.shape[0])
    cs = None if copy_stream is None else _stream(copy_stream)
    _check(lib().bergson_score_topk_host(
        _ptr(host_store), int(N), int(K), int(host_store.stride(0)), _ptr(queries), Q,
        int(queries.stride(0)), int(topk), 1 if least else 0, int(chunk_rows), _ptr(out_scores),
        _ptr(out_idx), _ptr(workspace), workspace.numel() * workspace.element_size(),
        _stream(stream), cs))


def bergson_token_scores_workspace(layers: Sequence, B: int, T: int, n_queries: int) -> int:
    arr = _layer_array(layers)
    n = ctypes.c_size_t()
    _check(lib().bergson_token_scores_workspace(arr, len(layers), int(B), int(T), int(n_queries),
                                                ctypes.byref(n)))
    return n.value


def bergson_token_scores(layers: Sequence, B: int, T: int, mask, queries, out, workspace,
                         stream=None) -> None:
    """Per-token scores out[q, b, t] of every token against each query row."""
    arr = _layer_array(layers)
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(lib().bergson_token_scores(arr, len(layers), int(B), int(T), _ptr(mask), _ptr(queries),
                                      int(queries.shape[0]), int(queries.stride(0)), _ptr(out),
                                      _ptr(workspace), ws_bytes, _stream(stream)))


def bergson_aggregate_rows_workspace(n: int) -> int:
    m = ctypes.c_size_t()
    _check(lib().bergson_aggregate_rows_workspace(int(n), ctypes.byref(m)))
    return m.value


def bergson_aggregate_rows(rows, n: int, K: int, offsets, mode: int, normalize_each: bool, out,
                           workspace=None, stream=None) -> None:
    """out[g] = sum/mean of rows[offsets[g]:offsets[g+1]] (offsets: device int64 [G+1])."""
    G = int(offsets.shape[0]) - 1
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib().bergson_aggregate_rows(_ptr(rows), int(n), int(K), int(rows.stride(0)),
                                        _ptr(offsets), G, int(mode), 1 if normalize_each else 0,
                                        _ptr(out), int(out.stride(0)), _ptr(workspace), ws_bytes,
                                        _stream(stream)))


def bergson_fisher_fit_workspace(n: int, K: int) -> int:
    m = ctypes.c_size_t()
    _check(lib().bergson_fisher_fit_workspace(int(n), int(K), ctypes.byref(m)))
    return m.value


def bergson_fisher_fit(rows, n: int, K: int, R, workspace, stream=None) -> None:
    """R = (1/n) sum_i rows[i] rows[i]^T (empirical Fisher of projected gradients)."""
    _check(lib().bergson_fisher_fit(_ptr(rows), int(n), int(K), int(rows.stride(0)), _ptr(R),
                                    int(R.stride(0)), _ptr(workspace),
                                    workspace.numel() * workspace.element_size(), _stream(stream)))


def bergson_fisher_preconditioner_workspace(K: int) -> int:
    m = ctypes.c_size_t()
    _check(lib().bergson_fisher_preconditioner_workspace(int(K), ctypes.byref(m)))
    return m.value


def bergson_fisher_preconditioner(R1, R2, K: int, lam: float, damping: float, power: int,
                                  iterations: int, M, workspace, stream=None) -> None:
    """M = (lam R1 + (1-lam) R2 + damping tr/K I)^-1/2 (or ^-1)."""
    _check(lib().bergson_fisher_preconditioner(
        _ptr(R1), _ptr(R2), int(K), int(R1.stride(0)), float(lam), float(damping), int(power),
        int(iterations), _ptr(M), int(M.stride(0)), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def bergson_fisher_preconditioner_tol(R1, R2, K: int, lam: float, damping: float, power: int,
                                      max_iterations: int, tol: float, M, workspace,
                                      stream=None) -> tuple[int, list]:
    """As bergson_fisher_preconditioner, stopping at the first iterate whose
    residual ||I - Z Y||_F / sqrt(K) is <= tol.  Returns (updates applied,
    residuals of the iterates computed)."""
    res = (ctypes.c_float * (int(max_iterations) + 1))(*([float("nan")] * (int(max_iterations) + 1)))
    done = ctypes.c_int()
    _check(lib().bergson_fisher_preconditioner_tol(
        _ptr(R1), _ptr(R2), int(K), int(R1.stride(0)), float(lam), float(damping), int(power),
        int(max_iterations), float(tol), _ptr(M), int(M.stride(0)), _ptr(workspace),
        workspace.numel() * workspace.element_size(), res, ctypes.byref(done), _stream(stream)))
    vals = [float(v) for v in res]
    return done.value, [v for v in vals if v == v]


def bergson_precondition_rows(rows, B: int, K: int, M, out, workspace, stream=None) -> None:
    """out[b] = M rows[b] (M symmetric K x K)."""
    _check(lib().bergson_precondition_rows(_ptr(rows), int(B), int(K), int(rows.stride(0)),
                                           _ptr(M), int(M.stride(0)), _ptr(out),
                                           int(out.stride(0)), _ptr(workspace),
                                           workspace.numel() * workspace.element_size(),
                                           _stream(stream)))


def bergson_store_save(store, rows: int, K: int, path: str, file_row_offset: int = 0,
                       stream=None) -> None:
    """Write device store rows [0, rows) to the raw fp16 store file at path."""
    _check(lib().bergson_store_save(_ptr(store), int(rows), int(K), int(store.stride(0)),
                                    os.fsencode(path), int(file_row_offset), _stream(stream)))


def bergson_store_load(path: str, file_row_offset: int, rows: int, K: int, store,
                       stream=None) -> None:
    """Read file rows [file_row_offset, +rows) into device store rows [0, rows)."""
    _check(lib().bergson_store_load(os.fsencode(path), int(file_row_offset), int(rows), int(K),
                                    _ptr(store), int(store.stride(0)), _stream(stream)))


def bergson_score_grads_workspace(B: int, K: int, Q: int) -> int:
    n = ctypes.c_size_t()
    _check(lib().bergson_score_grads_workspace(int(B), int(K), int(Q), ctypes.byref(n)))
    return n.value


def bergson_score_grads(proj, B: int, K: int, queries, unit_normalize: bool, scores, workspace,
                        stream=None) -> None:
    """On-the-fly scores of B projected rows against Q projected queries."""
    Q = int(queries.shape[0])
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(lib().bergson_score_grads(_ptr(proj), int(B), int(K), int(proj.stride(0)),
                                     _ptr(queries), Q, int(queries.stride(0)),
                                     1 if unit_normalize else 0, _ptr(scores),
                                     int(scores.stride(0)), _ptr(workspace), ws_bytes,
                                     _stream(stream)))


def bergson_projection_matrix(seed: int, d: int, k: int, proj_kind: int, moment, out,
                              stream=None) -> None:
    _check(lib().bergson_projection_matrix(int(seed), int(d), int(k), int(proj_kind), _ptr(moment),
                                           _ptr(out), _stream(stream)))


def bergson_sync_status(stream=None) -> int:
    """Returns the status code (does not raise)."""
    return lib().bergson_sync_status(_stream(stream))


def bergson_version() -> int:
    return lib().bergson_version()


def bergson_debug_wait_probe(timeout_ns: int, stream=None) -> None:
    _check(lib().bergson_debug_wait_probe(int(timeout_ns), _stream(stream)))


def bergson_debug_inject_status(status: int, count: int) -> None:
    lib().bergson_debug_inject_status(int(status), int(count))


def bergson_debug_attr_once(n_threads: int, n_devices: int, fail_device: int = -1):
    """(setting runs per simulated device, failed requests) of the per-device
    attribute record under n_threads concurrent first calls; host only."""
    calls = (ctypes.c_int64 * int(n_devices))()
    fails = ctypes.c_int()
    _check(lib().bergson_debug_attr_once(int(n_threads), int(n_devices), int(fail_device), calls,
                                         ctypes.byref(fails)))
    return list(calls), fails.value


def bergson_debug_project_plan(layers, B: int, T: int) -> tuple[int, int, int, int]:
    """(slots, work items, pieces, layers sharing their A) the projection planner
    chooses; host only."""
    arr = _layer_array(layers)
    n = [ctypes.c_int64() for _ in range(4)]
    _check(lib().bergson_debug_project_plan(arr, len(layers), int(B), int(T),
                                            *(ctypes.byref(x) for x in n)))
    return tuple(x.value for x in n)


SCORE_PLAN_COLUMNS = ("pass", "stage", "rows", "n_qg", "qg_base", "cpg", "grid", "n_tiles",
                      "q_begin", "q_end", "pair", "qt")


def bergson_debug_score_plan(N: int, K: int, Q: int, topk: int, ctas: int) -> list[dict]:
    """The score launches (one dict per launch, keys SCORE_PLAN_COLUMNS) the
    scorer's planner makes for `ctas` resident CTAs; host only."""
    n = ctypes.c_int32()
    _check(lib().bergson_debug_score_plan(int(N), int(K), int(Q), int(topk), int(ctas), None, 0,
                                          ctypes.byref(n)))
    buf = (ctypes.c_int64 * (12 * max(1, n.value)))()
    _check(lib().bergson_debug_score_plan(int(N), int(K), int(Q), int(topk), int(ctas), buf,
                                          n.value, ctypes.byref(n)))
    return [dict(zip(SCORE_PLAN_COLUMNS, buf[12 * i:12 * i + 12])) for i in range(n.value)]


XGEMM_PLAN_FIELDS = ("n_pad", "n_ntiles", "n_mtiles", "steps", "S", "stages", "n_chunks",
                     "pair", "n_buf", "y_rows", "tmem_cols", "xnorm_off", "ynorm_off",
                     "partial_off", "xh_off", "xl_off", "total", "a_base", "a_slots")


def bergson_debug_xgemm_plan(B: int, Q: int, K: int) -> dict:
    """The skinny-product planner's choices for B x rows, Q y rows, length K; host only."""
    buf = (ctypes.c_int64 * 19)()
    _check(lib().bergson_debug_xgemm_plan(int(B), int(Q), int(K), buf, 19))
    return dict(zip(XGEMM_PLAN_FIELDS, buf))


# ------------------------------------------------------------------ helpers

def workspace_tensor(nbytes: int, device="cuda"):
    """A byte tensor usable as workspace (torch allocations are 512-byte aligned)."""
    import torch
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)
