"""GB300-native ARC-KV per-context KV-cache compaction.

A thin ctypes binding over ``libarckv.so`` (C ABI in ``include/arckv.h``).
The functions here only marshal arguments: every step of the compaction
runs in the library's CUDA kernels for sm_103a.  PyTorch tensors are used for
device memory and streams.  There is no CPU fallback: if the library is not
built, every call raises.
"""
from __future__ import annotations

import ctypes
import dataclasses
from pathlib import Path
from typing import Dict, Optional, Sequence

__all__ = [
    "Config", "ArckvError", "STATUS", "NUM_STAGES", "STAGE_NAMES", "load_library", "workspace_bytes", "anchor_count",
    "attend_workspace_bytes", "arckv_compact", "arckv_attend", "arckv_query_status", "status_string",
    "compact_layer", "attend", "INDEXER_FIELDS", "attend_joint", "arckv_attend_joint",
    "attend_joint_workspace_bytes", "FLAG_COMPACT_BF16", "truncated_error", "arckv_truncated_error", "SELECTOR_INDEXER", "SELECTOR_HA", "SELECTOR_VI",
    "arckv_wait_probe",
]

_LIB_PATH = Path(__file__).resolve().parent / "libarckv.so"
_lib = None

STATUS = {
    0: "ARCKV_OK", 1: "ARCKV_ERR_INVALID_ARG", 2: "ARCKV_ERR_SHAPE", 3: "ARCKV_ERR_WORKSPACE",
    4: "ARCKV_ERR_NOT_SPD", 5: "ARCKV_ERR_NONFINITE", 6: "ARCKV_ERR_TIMEOUT", 7: "ARCKV_ERR_CUDA",
    8: "ARCKV_ERR_UNSUPPORTED",
}
FLAG_NONBLOCKING = 0x1
FLAG_COMPACT_BF16 = 0x2
SELECTOR_INDEXER, SELECTOR_HA, SELECTOR_VI = 0, 1, 2
NUM_STAGES = 11
STAGE_NAMES = ("indexer_features", "index_logits", "pool_top_t", "reference_attention", "column_profiles",
               "assignment", "merge", "beta_products", "beta_solve", "value_products", "value_solve")
INDEXER_FIELDS = ("L_q", "L_k", "L_x", "b_x", "U_q", "U_k", "U_v", "L_c", "L_v")


class ArckvError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__("%s: %s (%s)" % (where, STATUS.get(code, code), status_string(code)))


class _Config(ctypes.Structure):
    _fields_ = ([(n, ctypes.c_int32) for n in
                 ("H_kv", "G", "T", "d", "n_pos", "d_x", "H_I", "d_I", "d_A", "t", "chunk_len")] +
                [(n, ctypes.c_float) for n in
                 ("lambda_m", "logit_scale", "ridge_w", "ridge_v", "eps_w", "b_min", "b_max")] +
                [("flags", ctypes.c_uint32), ("selector", ctypes.c_int32)])


class _Indexer(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in INDEXER_FIELDS]


class _Aux(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("scores", "anchors", "assign", "anchors_in", "assign_in", "stage_events", "launches")]


@dataclasses.dataclass
class Config:
    """One layer's compaction problem (mirrors ``arckv_config``)."""
    H_kv: int
    T: int
    n_pos: int
    t: int
    G: int = 4
    d: int = 128
    d_x: int = 4096
    H_I: int = 8
    d_I: int = 128
    d_A: int = 128
    chunk_len: int = 0
    lambda_m: float = 0.25
    logit_scale: float = 0.0
    ridge_w: float = 1e-4
    ridge_v: float = 1e-3
    eps_w: float = 2.0611536e-09  # e^-20
    b_min: float = -20.0
    b_max: float = 20.0
    flags: int = 0
    selector: int = 0             # SELECTOR_INDEXER / SELECTOR_HA / SELECTOR_VI (App. B.1)

    @property
    def n(self) -> int:
        return self.n_pos * self.G

    def c_struct(self) -> _Config:
        return _Config(self.H_kv, self.G, self.T, self.d, self.n_pos, self.d_x, self.H_I, self.d_I, self.d_A,
                       self.t, self.chunk_len, self.lambda_m, self.logit_scale, self.ridge_w, self.ridge_v,
                       self.eps_w, self.b_min, self.b_max, self.flags, self.selector)


def load_library():
    """Load libarckv.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not _LIB_PATH.exists():
        raise RuntimeError("%s is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`"
                           % _LIB_PATH)
    lib = ctypes.CDLL(str(_LIB_PATH))
    P = ctypes.c_void_p
    lib.arckv_workspace_bytes.argtypes = [ctypes.POINTER(_Config)]
    lib.arckv_workspace_bytes.restype = ctypes.c_size_t
    lib.arckv_anchor_count.argtypes = [ctypes.POINTER(_Config)]
    lib.arckv_anchor_count.restype = ctypes.c_int32
    lib.arckv_compact.argtypes = [ctypes.POINTER(_Config), P, P, P, P, ctypes.POINTER(_Indexer), P, P, P,
                                  ctypes.POINTER(_Aux), P, ctypes.c_size_t, P]
    lib.arckv_compact.restype = ctypes.c_int
    lib.arckv_attend_workspace_bytes.argtypes = [ctypes.c_int32] * 4
    lib.arckv_attend_workspace_bytes.restype = ctypes.c_size_t
    lib.arckv_attend.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_float,
                                 P, P, P, P, P, P, ctypes.c_size_t, ctypes.c_uint32, P]
    lib.arckv_attend.restype = ctypes.c_int
    lib.arckv_attend_joint_workspace_bytes.argtypes = [ctypes.c_int32] * 5
    lib.arckv_attend_joint_workspace_bytes.restype = ctypes.c_size_t
    lib.arckv_attend_joint.argtypes = [ctypes.c_int32] * 5 + [ctypes.c_float] + [P] * 8 + [ctypes.c_size_t,
                                                                                         ctypes.c_uint32, P]
    lib.arckv_attend_joint.restype = ctypes.c_int
    lib.arckv_truncated_error_workspace_bytes.argtypes = [ctypes.c_int32] * 5
    lib.arckv_truncated_error_workspace_bytes.restype = ctypes.c_size_t
    lib.arckv_truncated_error.argtypes = [ctypes.c_int32] * 5 + [ctypes.c_float] + [P] * 5 + [P, ctypes.c_size_t,
                                                                                              ctypes.c_uint32, P]
    lib.arckv_truncated_error.restype = ctypes.c_int
    lib.arckv_query_status.argtypes = [P, P]
    lib.arckv_query_status.restype = ctypes.c_int
    lib.arckv_wait_probe.argtypes = [P, ctypes.c_size_t, ctypes.c_uint32, P]
    lib.arckv_wait_probe.restype = ctypes.c_int
    lib.arckv_status_string.argtypes = [ctypes.c_int]
    lib.arckv_status_string.restype = ctypes.c_char_p
    _lib = lib
    return lib


def status_string(code: int) -> str:
    return load_library().arckv_status_string(int(code)).decode()


def workspace_bytes(cfg: Config) -> int:
    c = cfg.c_struct()
    return int(load_library().arckv_workspace_bytes(ctypes.byref(c)))


def anchor_count(cfg: Config) -> int:
    """Realized anchors per head t' (App. A.3 chunking; = cfg.t without it), 0 if invalid."""
    c = cfg.c_struct()
    return int(load_library().arckv_anchor_count(ctypes.byref(c)))


def attend_workspace_bytes(H_kv: int, n: int, t: int, d: int = 128) -> int:
    return int(load_library().arckv_attend_workspace_bytes(H_kv, n, t, d))


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if not x.is_contiguous():
        # the C ABI takes dense row-major arrays; a strided view would be read with the wrong layout
        raise ValueError("arckv: tensor arguments must be contiguous (row-major); got strides %s"
                         % (tuple(x.stride()),))
    return x.data_ptr()


def _expect(name: str, x, dtypes, shape=None):
    """Check a torch tensor argument of the helpers below: dtype, shape (None
    entries match any extent) and dense layout.  Raises ValueError."""
    import torch
    if not isinstance(x, torch.Tensor):
        raise ValueError("arckv: %s must be a torch tensor" % name)
    if x.dtype not in dtypes:
        raise ValueError("arckv: %s must be %s, got %s" % (name, " or ".join(map(str, dtypes)), x.dtype))
    if shape is not None and (x.dim() != len(shape) or
                              any(w is not None and int(g) != int(w) for g, w in zip(x.shape, shape))):
        raise ValueError("arckv: %s must have shape %s, got %s" % (
            name, tuple("*" if w is None else w for w in shape), tuple(x.shape)))
    if not x.is_contiguous():
        raise ValueError("arckv: %s must be contiguous (row-major)" % name)


def _on_one_cuda_device(**tensors):
    """All given tensors (None entries skipped) on one CUDA device: the
    kernels read them there and there is no CPU path.  Raises ValueError."""
    dev = None
    for name, x in tensors.items():
        if x is None:
            continue
        if x.device.type != "cuda":
            raise ValueError("arckv: %s must be on a CUDA device, got %s (there is no CPU path)" % (name, x.device))
        if dev is not None and x.device != dev:
            raise ValueError("arckv: %s is on %s but the other arguments on %s" % (name, x.device, dev))
        dev = x.device


def _stream_handle(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def arckv_compact(cfg: Config, K, V, Q_ref, X_ref, idx: Dict[str, object], C_k, beta, C_v, ws, ws_bytes: int,
                  stream=None, scores=None, anchors=None, assign=None, anchors_in=None, assign_in=None,
                  stage_events: Optional[Sequence[int]] = None):
    """Direct binding of ``arckv_compact``.  Tensor arguments may be torch
    tensors or raw device addresses.  Returns (status, launches)."""
    lib = load_library()
    c = cfg.c_struct()
    ix = _Indexer(*[_ptr(idx.get(n)) if idx is not None else None for n in INDEXER_FIELDS])
    launches = ctypes.c_int32(0)
    ev_arr = None
    if stage_events is not None:
        ev_arr = (ctypes.c_void_p * len(stage_events))(*stage_events)
    aux = _Aux(_ptr(scores), _ptr(anchors), _ptr(assign), _ptr(anchors_in), _ptr(assign_in),
               ctypes.cast(ev_arr, ctypes.c_void_p) if ev_arr is not None else None,
               ctypes.cast(ctypes.pointer(launches), ctypes.c_void_p))
    st = lib.arckv_compact(ctypes.byref(c), _ptr(K), _ptr(V), _ptr(Q_ref), _ptr(X_ref), ctypes.byref(ix),
                           _ptr(C_k), _ptr(beta), _ptr(C_v), ctypes.byref(aux), _ptr(ws), int(ws_bytes),
                           _stream_handle(stream))
    return int(st), int(launches.value)


def arckv_attend(H_kv: int, n: int, t: int, d: int, logit_scale: float, Q, C_k, beta, C_v, O, ws, ws_bytes: int,
                 flags: int = 0, stream=None) -> int:
    """Direct binding of ``arckv_attend``; returns the status code."""
    lib = load_library()
    return int(lib.arckv_attend(H_kv, n, t, d, float(logit_scale), _ptr(Q), _ptr(C_k), _ptr(beta), _ptr(C_v),
                                _ptr(O), _ptr(ws), int(ws_bytes), int(flags), _stream_handle(stream)))


def attend_joint_workspace_bytes(H: int, n: int, t: int, F: int, d: int = 128) -> int:
    return int(load_library().arckv_attend_joint_workspace_bytes(H, n, t, F, d))


def arckv_attend_joint(H: int, n: int, t: int, F: int, d: int, logit_scale: float, Q, C_k, beta, C_v, K_fixed,
                       V_fixed, O, ws, ws_bytes: int, flags: int = 0, stream=None) -> int:
    """Direct binding of ``arckv_attend_joint``; returns the status code."""
    lib = load_library()
    return int(lib.arckv_attend_joint(H, n, t, F, d, float(logit_scale), _ptr(Q), _ptr(C_k), _ptr(beta), _ptr(C_v),
                                      _ptr(K_fixed), _ptr(V_fixed), _ptr(O), _ptr(ws), int(ws_bytes), int(flags),
                                      _stream_handle(stream)))


def arckv_truncated_error(H: int, n: int, T: int, t: int, d: int, logit_scale: float, Q_eval, K, V, S, E, ws,
                          ws_bytes: int, flags: int = 0, stream=None) -> int:
    """Direct binding of ``arckv_truncated_error``; returns the status code."""
    lib = load_library()
    return int(lib.arckv_truncated_error(H, n, T, t, d, float(logit_scale), _ptr(Q_eval), _ptr(K), _ptr(V), _ptr(S),
                                         _ptr(E), _ptr(ws), int(ws_bytes), int(flags), _stream_handle(stream)))


def arckv_query_status(ws, stream=None) -> int:
    return int(load_library().arckv_query_status(_ptr(ws), _stream_handle(stream)))


def arckv_wait_probe(ws, ws_bytes: int, limit_us: int, stream=None) -> int:
    """Direct binding of ``arckv_wait_probe`` (a bounded device wait made to
    give up); returns the status code."""
    return int(load_library().arckv_wait_probe(_ptr(ws), int(ws_bytes), int(limit_us), _stream_handle(stream)))


# ----------------------------------------------------------- torch helpers

def _alloc_ws(nbytes: int, device):
    import torch
    return torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)


def compact_layer(cfg: Config, K, V, Q_ref, X_ref, idx: Dict[str, object], *, ws=None, anchors_in=None,
                  assign_in=None, want_scores: bool = False, want_anchors: bool = True,
                  want_assign: bool = False, stream=None, stage_events=None, check: bool = True):
    """Allocate outputs (and a workspace unless given) with torch on K's device
    and call ``arckv_compact``.  Returns a dict of tensors plus 'status' and
    'launches'.  Raises ArckvError on a non-OK status when ``check``."""
    import torch
    bf, i32 = (torch.bfloat16,), (torch.int32,)
    H, T, d, n = cfg.H_kv, cfg.T, cfg.d, cfg.n_pos * cfg.G
    _expect("K", K, bf, (H, T, d))
    _expect("V", V, bf, (H, T, d))
    _expect("Q_ref", Q_ref, bf)
    if Q_ref.shape[0] != H or Q_ref.numel() != H * n * d:
        raise ValueError("arckv: Q_ref must hold [H_kv][n_pos * G][d] = %s, got shape %s"
                         % ((H, n, d), tuple(Q_ref.shape)))
    if cfg.selector == SELECTOR_INDEXER and anchors_in is None:
        _expect("X_ref", X_ref, bf, (cfg.n_pos, cfg.d_x))
        for f in INDEXER_FIELDS:
            _expect("indexer." + f, idx.get(f), bf)
            if idx[f].shape[0] != H:
                raise ValueError("arckv: indexer.%s must lead with H_kv = %d, got shape %s"
                                 % (f, H, tuple(idx[f].shape)))
    if anchors_in is not None:
        _expect("anchors_in", anchors_in, i32, (H, anchor_count(cfg)))
    if assign_in is not None:
        _expect("assign_in", assign_in, i32, (H, T))
    checked_idx = {} if not (cfg.selector == SELECTOR_INDEXER and anchors_in is None) else \
        {"X_ref": X_ref, **{"indexer." + f: idx[f] for f in INDEXER_FIELDS}}
    _on_one_cuda_device(K=K, V=V, Q_ref=Q_ref, anchors_in=anchors_in, assign_in=assign_in, **checked_idx)
    dev = K.device
    f32 = dict(dtype=torch.float32, device=dev)
    need = workspace_bytes(cfg)
    if need == 0:
        raise ArckvError(2, "arckv_workspace_bytes")
    if ws is None:
        ws = _alloc_ws(need, dev)
    tp = anchor_count(cfg)
    out = {
        "C_k": torch.empty(cfg.H_kv, tp, cfg.d, **f32),
        "beta": torch.empty(cfg.H_kv, tp, **f32),
        "C_v": torch.empty(cfg.H_kv, tp, cfg.d, **f32),
    }
    if want_scores:
        out["scores"] = torch.empty(cfg.H_kv, cfg.T, **f32)
    if want_anchors:
        out["anchors"] = torch.empty(cfg.H_kv, tp, dtype=torch.int32, device=dev)
    if want_assign:
        out["assign"] = torch.empty(cfg.H_kv, cfg.T, dtype=torch.int32, device=dev)
    st, nl = arckv_compact(cfg, K, V, Q_ref, X_ref, idx, out["C_k"], out["beta"], out["C_v"], ws, ws.numel(),
                           stream=stream, scores=out.get("scores"), anchors=out.get("anchors"),
                           assign=out.get("assign"), anchors_in=anchors_in, assign_in=assign_in,
                           stage_events=stage_events)
    if check and st != 0:
        raise ArckvError(st, "arckv_compact")
    out["status"], out["launches"] = st, nl
    return out


def attend(Q, C_k, beta, C_v, logit_scale: float = 0.0, *, ws=None, stream=None, check: bool = True):
    """O = softmax(scale Q C_k^T + beta) C_v for Q [H, n, 128] bf16 on the device."""
    import torch
    _expect("Q", Q, (torch.bfloat16,), (None, None, None))
    H, n, d = Q.shape
    _expect("C_k", C_k, (torch.float32,), (H, None, d))
    t = C_k.shape[1]
    _expect("beta", beta, (torch.float32,), (H, t))
    _expect("C_v", C_v, (torch.float32,), (H, t, d))
    _on_one_cuda_device(Q=Q, C_k=C_k, beta=beta, C_v=C_v)
    need = attend_workspace_bytes(H, n, t, d)
    if need == 0:
        raise ArckvError(2, "arckv_attend_workspace_bytes")
    if ws is None:
        ws = _alloc_ws(need, Q.device)
    O = torch.empty(H, n, d, dtype=torch.float32, device=Q.device)
    st = arckv_attend(H, n, t, d, logit_scale, Q, C_k, beta, C_v, O, ws, ws.numel(), stream=stream)
    if check and st != 0:
        raise ArckvError(st, "arckv_attend")
    return O


def attend_joint(Q, C_k=None, beta=None, C_v=None, K_fixed=None, V_fixed=None, logit_scale: float = 0.0, *, ws=None,
                 stream=None, check: bool = True):
    """O = softmax(scale Q [C_k; K_fixed]^T + [beta; 0]) [C_v; V_fixed] (App. A.7) for Q [H, n, 128] bf16.
    C_k / C_v fp32 or bf16 (both the same); either block may be omitted."""
    import torch
    _expect("Q", Q, (torch.bfloat16,), (None, None, None))
    H, n, d = Q.shape
    if (C_k is None) != (C_v is None) or (C_k is None) != (beta is None):
        raise ValueError("arckv: C_k, beta and C_v are given together or not at all")
    if (K_fixed is None) != (V_fixed is None):
        raise ValueError("arckv: K_fixed and V_fixed are given together or not at all")
    if C_k is not None:
        _expect("C_k", C_k, (torch.float32, torch.bfloat16), (H, None, d))
        _expect("C_v", C_v, (C_k.dtype,), (H, C_k.shape[1], d))
        _expect("beta", beta, (torch.float32,), (H, C_k.shape[1]))
    if K_fixed is not None:
        _expect("K_fixed", K_fixed, (torch.bfloat16,), (H, None, d))
        _expect("V_fixed", V_fixed, (torch.bfloat16,), (H, K_fixed.shape[1], d))
    _on_one_cuda_device(Q=Q, C_k=C_k, beta=beta, C_v=C_v, K_fixed=K_fixed, V_fixed=V_fixed)
    t = 0 if C_k is None else C_k.shape[1]
    F = 0 if K_fixed is None else K_fixed.shape[1]
    need = attend_joint_workspace_bytes(H, n, t, F, d)
    if need == 0:
        raise ArckvError(2, "arckv_attend_joint_workspace_bytes")
    if ws is None:
        ws = _alloc_ws(need, Q.device)
    flags = FLAG_COMPACT_BF16 if (C_k is not None and C_k.dtype == torch.bfloat16) else 0
    O = torch.empty(H, n, d, dtype=torch.float32, device=Q.device)
    st = arckv_attend_joint(H, n, t, F, d, logit_scale, Q, C_k, beta, C_v, K_fixed, V_fixed, O, ws, ws.numel(),
                            flags=flags, stream=stream)
    if check and st != 0:
        raise ArckvError(st, "arckv_attend_joint")
    return O


def truncated_error(Q_eval, K, V, S, logit_scale: float = 0.0, *, stream=None, check: bool = True):
    """E(S) per head (App. B.1) for Q_eval [H, n, 128], K, V [H, T, 128] bf16 and anchors S [H, t] int32."""
    import torch
    _expect("Q_eval", Q_eval, (torch.bfloat16,), (None, None, None))
    H, n, d = Q_eval.shape
    _expect("K", K, (torch.bfloat16,), (H, None, d))
    T = K.shape[1]
    _expect("V", V, (torch.bfloat16,), (H, T, d))
    if S is not None:
        _expect("S", S, (torch.int32,), (H, None))
    _on_one_cuda_device(Q_eval=Q_eval, K=K, V=V, S=S)
    t = 0 if S is None else S.shape[1]
    need = int(load_library().arckv_truncated_error_workspace_bytes(H, n, T, t, d))
    if need == 0:
        raise ArckvError(2, "arckv_truncated_error_workspace_bytes")
    ws = _alloc_ws(need, Q_eval.device)
    E = torch.empty(H, dtype=torch.float32, device=Q_eval.device)
    st = arckv_truncated_error(H, n, T, t, d, logit_scale, Q_eval, K, V, S, E, ws, ws.numel(), stream=stream)
    if check and st != 0:
        raise ArckvError(st, "arckv_truncated_error")
    return E
