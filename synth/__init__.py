"""Seeded synthetic inputs for per-context KV-cache compaction.

This module is shared by the fp64 oracle (``oracle/``) and by the CUDA path
(``paper_2609_36835_gb300``).  It holds only the input recipe -- random
draws, RoPE of the synthetic keys, bf16 rounding -- and none of the
compaction arithmetic.  Every tensor is produced on the host from a
counter-based Philox-4x32-10 stream (Salmon et al., SC'11, as implemented by
``numpy.random.Philox``) keyed by (workload, layer, KV head, stream id), so
any single (layer, head) pair can be regenerated on its own.

Recipe (stands in for the repeat-prefilled Llama-3.1-8B caches of the paper's
evaluation, which are not available; Sec. 3.1, App. A.1, App. A.5):

* keys: N(0,1)^{T x d}; 4 seeded channels multiplied by 8 (outlier channels),
  then Llama rotate-half RoPE with theta = 500000 at positions 0..T-1, then
  row 0 scaled to 10x its norm (attention sink);
* values: N(0,1)^{T x d}, no rotation;
* reference queries (n_q = n_pos * G rows per KV head, row i = r*G + g):
  a uniformly drawn key plus N(0, 0.5^2) noise;
* reference activations x_r: N(0,1)^{d_x}, one per reference position,
  shared by the G query heads of that position and by all KV heads of a layer;
* held-out queries: same law as the reference queries, separate stream;
* stand-in compact caches for attention tests (no fit involved): C_k = the
  keys at a uniformly drawn anchor subset plus N(0, 0.1^2) noise, C_v = the
  values there, beta ~ U(-2, 1);
* decode batches (timing and full-size attention parity): keys, values and
  queries N(0,1) in bf16 drawn on the device by a seeded torch generator
  (Philox on CUDA), stand-in compact caches drawn the same way;
* whole layers for timing (``make_layer_device``): the same recipe for K, V
  and Q_ref, drawn by a seeded torch generator on the device (a different
  random stream from the host path, the same distributions), so that a 32-layer
  128K context is generated in seconds; X_ref and the indexer weights come from
  the host path;
* indexer weights in the shapes of Eqs. (indexer_parameters) and
  (value_indexer_parameters): U_q, U_k, U_v, L_q, L_k, L_v ~ N(0, 1/d),
  L_c ~ N(0, 1/d_A), L_x ~ N(0, 1/d_x), b_x ~ N(0, 0.1^2).

All tensors are returned as bf16 bit patterns (``numpy.uint16``); the oracle
widens them exactly to float64 and the GPU path uploads the same bytes.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Optional

import numpy as np

__all__ = [
    "Workload", "WORKLOADS", "IndexerShape", "bf16_round", "bf16_to_f64",
    "bf16_to_f32", "make_pair", "make_layer_activations", "make_heldout",
    "make_indexer", "make_compact_cache", "decode_batch_device", "make_layer_device",
]

D_HEAD = 128
ROPE_THETA = 500000.0


@dataclasses.dataclass(frozen=True)
class IndexerShape:
    """Widths of one layer-KV-head indexer (App. A.1)."""
    d: int = D_HEAD       # model head dim
    d_x: int = 4096       # pre-query-projection activation width (Llama hidden)
    H_I: int = 8          # index heads
    d_I: int = 128        # index head width
    d_A: int = 128        # value-attention head width


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic compaction workload (a context of ``layers`` x ``H_kv`` pairs)."""
    name: str
    wid: int              # seed component
    layers: int
    H_kv: int
    T: int
    n_pos: int            # reference positions; rows per KV head n = n_pos * G
    t: int
    G: int = 4
    outliers_per_layer: bool = False
    shape: IndexerShape = IndexerShape()

    @property
    def n(self) -> int:
        return self.n_pos * self.G


WORKLOADS: Dict[str, Workload] = {
    # single head group, one layer
    "single_head_T1024": Workload("single_head_T1024", 0, 1, 1, 1024, 64, 102),
    # one Llama-3.1-8B layer
    "llama8b_layer_T8192": Workload("llama8b_layer_T8192", 1, 1, 8, 8192, 256, 819),
    # the full 32-layer Llama-3.1-8B cache at three retentions (suffix rNN: t / T = NN %)
    "llama8b_T8192_r10": Workload("llama8b_T8192_r10", 2, 32, 8, 8192, 256, 819),
    "llama8b_T8192_r05": Workload("llama8b_T8192_r05", 2, 32, 8, 8192, 256, 409),
    "llama8b_T8192_r02": Workload("llama8b_T8192_r02", 2, 32, 8, 8192, 256, 163),
    # 32K context, outlier channels reseeded per layer
    "llama8b_T32768_r05": Workload("llama8b_T32768_r05", 3, 32, 8, 32768, 512, 1638,
                                   outliers_per_layer=True),
    # 128K context, large t x t fits
    "llama8b_T131072_r10": Workload("llama8b_T131072_r10", 4, 32, 8, 131072, 512, 13107),
}

# stream ids (one Philox key per tensor family)
_S_KEYS, _S_VALS, _S_QREF, _S_XREF, _S_HOLD, _S_IDX, _S_OUTL, _S_CCACHE = range(1, 9)


def _rng(*key: int) -> np.random.Generator:
    ss = np.random.SeedSequence([0xA2C4, *[int(k) for k in key]])
    return np.random.Generator(np.random.Philox(ss))


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (round to nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_to_f32(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << 16).view(np.float32)


def bf16_to_f64(b: np.ndarray) -> np.ndarray:
    return bf16_to_f32(b).astype(np.float64)


def _rope(x: np.ndarray, positions: np.ndarray, theta: float = ROPE_THETA) -> np.ndarray:
    """Llama rotate-half RoPE on rows of x (float64), pairing channel i with i + d/2."""
    d = x.shape[-1]
    half = d // 2
    inv_freq = theta ** (-np.arange(half, dtype=np.float64) * 2.0 / d)
    ang = positions[:, None].astype(np.float64) * inv_freq[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[:, :half], x[:, half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=1)


def _outlier_channels(w: Workload, layer: int) -> np.ndarray:
    g = _rng(w.wid, layer if w.outliers_per_layer else 0, 0, _S_OUTL)
    return np.sort(g.choice(D_HEAD, size=4, replace=False))


def _keys(w: Workload, layer: int, head: int, T: Optional[int] = None) -> np.ndarray:
    T = w.T if T is None else T
    g = _rng(w.wid, layer, head, _S_KEYS)
    k = g.standard_normal((T, D_HEAD))
    k[:, _outlier_channels(w, layer)] *= 8.0
    k = _rope(k, np.arange(T))
    k[0] *= 10.0
    return bf16_round(k.astype(np.float32))


def _queries_like_keys(keys_bf16: np.ndarray, n: int, g: np.random.Generator) -> np.ndarray:
    T = keys_bf16.shape[0]
    j = g.integers(0, T, size=n)
    q = bf16_to_f64(keys_bf16[j]) + 0.5 * g.standard_normal((n, D_HEAD))
    return bf16_round(q.astype(np.float32))


def make_indexer(w: Workload, layer: int, head: int, zero_value_path: bool = False) -> Dict[str, np.ndarray]:
    """Seeded indexer parameters of one (layer, KV head) pair, bf16 bits.

    Shapes follow App. A.1: L_q, L_k, L_c, L_v are [H_I*d_I, *]; L_x is
    [H_I, d_x]; b_x is [H_I]; U_q, U_k, U_v are [d_A, d].  With
    ``zero_value_path`` the value pathway L_c, L_v is zero (the paper's
    initialisation, under which the logits do not depend on V).
    """
    s = w.shape
    g = _rng(w.wid, layer, head, _S_IDX)
    HD = s.H_I * s.d_I

    def nrm(shape, std):
        return bf16_round((std * g.standard_normal(shape)).astype(np.float32))

    p = {
        "U_q": nrm((s.d_A, s.d), s.d ** -0.5),
        "U_k": nrm((s.d_A, s.d), s.d ** -0.5),
        "U_v": nrm((s.d_A, s.d), s.d ** -0.5),
        "L_q": nrm((HD, s.d), s.d ** -0.5),
        "L_k": nrm((HD, s.d), s.d ** -0.5),
        "L_v": nrm((HD, s.d), s.d ** -0.5),
        "L_c": nrm((HD, s.d_A), s.d_A ** -0.5),
        "L_x": nrm((s.H_I, s.d_x), s.d_x ** -0.5),
        "b_x": nrm((s.H_I,), 0.1),
    }
    if zero_value_path:
        p["L_c"] = np.zeros_like(p["L_c"])
        p["L_v"] = np.zeros_like(p["L_v"])
    return p


def make_layer_activations(w: Workload, layer: int, n_pos: Optional[int] = None) -> np.ndarray:
    """X_ref of one layer: [n_pos, d_x] bf16 bits, shared by all KV heads."""
    n_pos = w.n_pos if n_pos is None else n_pos
    g = _rng(w.wid, layer, 0, _S_XREF)
    return bf16_round(g.standard_normal((n_pos, w.shape.d_x)).astype(np.float32))


def make_pair(w: Workload, layer: int, head: int, T: Optional[int] = None,
              n_pos: Optional[int] = None) -> Dict[str, np.ndarray]:
    """K, V [T, d] and Q_ref [n, d] (row i = r*G + g) of one pair, bf16 bits.

    ``T`` / ``n_pos`` override the workload's sizes (used for small test cases
    that keep the workload's distributions).
    """
    T = w.T if T is None else T
    n_pos = w.n_pos if n_pos is None else n_pos
    K = _keys(w, layer, head, T)
    gv = _rng(w.wid, layer, head, _S_VALS)
    V = bf16_round(gv.standard_normal((T, D_HEAD)).astype(np.float32))
    gq = _rng(w.wid, layer, head, _S_QREF)
    Q = _queries_like_keys(K, n_pos * w.G, gq)
    return {"K": K, "V": V, "Q": Q}


def make_heldout(w: Workload, layer: int, head: int, K_bf16: np.ndarray, n: int) -> np.ndarray:
    """Held-out queries (same law as Q_ref, separate stream): [n, d] bf16 bits."""
    return _queries_like_keys(K_bf16, n, _rng(w.wid, layer, head, _S_HOLD))


def make_compact_cache(w: Workload, layer: int, head: int, K_bf16: np.ndarray, V_bf16: np.ndarray,
                       t: int) -> Dict[str, np.ndarray]:
    """A stand-in compact cache of t rows (fp32) for attention tests: the
    keys at t distinct random positions plus N(0, 0.1^2) noise, the values
    there, beta ~ U(-2, 1).  No part of the compaction method is involved."""
    g = _rng(w.wid, layer, head, _S_CCACHE)
    S = np.sort(g.choice(K_bf16.shape[0], size=t, replace=False))
    C_k = (bf16_to_f64(K_bf16[S]) + 0.1 * g.standard_normal((t, D_HEAD))).astype(np.float32)
    C_v = bf16_to_f64(V_bf16[S]).astype(np.float32)
    beta = g.uniform(-2.0, 1.0, size=t).astype(np.float32)
    return {"C_k": C_k, "C_v": C_v, "beta": beta}


def decode_batch_device(seed: int, H: int, G: int, T: int, t: int, F: int, device, compact_bf16: bool = True):
    """One decode step's inputs on the device, drawn by a seeded torch
    generator: Q [H, G, d], full cache K, V [H, T, d] and an uncompressed block
    K_f, V_f [H, F, d] (bf16, N(0,1)); a stand-in compact cache C_k, C_v
    [H, t, d] (bf16 or fp32, N(0,1)) and beta [H, t] ~ U(-2, 1)."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    def nrm(*shape, dt=torch.bfloat16):
        return torch.randn(*shape, generator=gen, device=device, dtype=torch.float32).to(dt)
    cdt = torch.bfloat16 if compact_bf16 else torch.float32
    out = {"Q": nrm(H, G, D_HEAD), "K": nrm(H, T, D_HEAD), "V": nrm(H, T, D_HEAD),
           "C_k": nrm(H, t, D_HEAD, dt=cdt), "C_v": nrm(H, t, D_HEAD, dt=cdt),
           "beta": torch.rand(H, t, generator=gen, device=device) * 3.0 - 2.0,
           "K_f": nrm(H, F, D_HEAD), "V_f": nrm(H, F, D_HEAD)}
    return out


def _torch_seed(*key: int) -> int:
    """A 63-bit torch seed derived from the same key as the host streams."""
    ss = np.random.SeedSequence([0xA2C4, *[int(k) for k in key]])
    return int(ss.generate_state(2, dtype=np.uint32).astype(np.uint64) @ np.array([1, 1 << 32], dtype=np.uint64)
               & np.uint64((1 << 63) - 1))


def _rope_torch(x, positions, theta: float = ROPE_THETA):
    """_rope on a torch tensor: rotation angles in float64, applied in float32."""
    import torch
    d = x.shape[-1]
    half = d // 2
    inv_freq = theta ** (-torch.arange(half, dtype=torch.float64, device=x.device) * 2.0 / d)
    ang = positions[:, None].to(torch.float64) * inv_freq[None, :]
    c, s_ = torch.cos(ang).to(torch.float32), torch.sin(ang).to(torch.float32)
    lo, hi = x[:, :half], x[:, half:]   # rotate-half pairs (i, i + d/2)
    return torch.cat([lo * c - hi * s_, hi * c + lo * s_], dim=1)


def make_layer_device(w: Workload, layer: int, heads, device, T: Optional[int] = None, n_pos: Optional[int] = None):
    """One layer's inputs as torch tensors on ``device``: K, V [H][T][d] and
    Q_ref [H][n][d] (bf16) drawn by the recipe above from a seeded torch
    generator per (layer, head); X [n_pos][d_x] and the indexer fields
    [H][...] (bf16) from the host path.  Row i of Q_ref is r*G + g."""
    import torch
    T = w.T if T is None else T
    n_pos = w.n_pos if n_pos is None else n_pos
    n = n_pos * w.G
    Ks, Vs, Qs = [], [], []
    for h in heads:
        g = torch.Generator(device=device)
        g.manual_seed(_torch_seed(w.wid, layer, h, _S_KEYS))
        k = torch.randn(T, D_HEAD, generator=g, device=device, dtype=torch.float32)
        k[:, torch.as_tensor(_outlier_channels(w, layer), device=device)] *= 8.0
        k = _rope_torch(k, torch.arange(T, device=device))
        k[0] = k[0] * 10.0
        kb = k.to(torch.bfloat16)
        g.manual_seed(_torch_seed(w.wid, layer, h, _S_VALS))
        vb = torch.randn(T, D_HEAD, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
        g.manual_seed(_torch_seed(w.wid, layer, h, _S_QREF))
        j = torch.randint(0, T, (n,), generator=g, device=device)
        q = kb[j].to(torch.float32) + 0.5 * torch.randn(n, D_HEAD, generator=g, device=device, dtype=torch.float32)
        Ks.append(kb)
        Vs.append(vb)
        Qs.append(q.to(torch.bfloat16))
        del k
    out = {"K": torch.stack(Ks), "V": torch.stack(Vs), "Q": torch.stack(Qs)}

    def host_bits(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)

    out["X"] = host_bits(make_layer_activations(w, layer, n_pos=n_pos))
    idx = [make_indexer(w, layer, h) for h in heads]
    for f in idx[0]:
        out[f] = host_bits(np.stack([ix[f] for ix in idx]))
    return out
