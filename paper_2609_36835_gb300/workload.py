"""Stack seeded synthetic inputs (``synth``) into the layer tensors that
``arckv_compact`` takes.  Marshalling only: bf16 bit patterns are copied
unchanged into torch tensors."""
from __future__ import annotations

from typing import Dict, Optional, Sequence

import numpy as np

import synth

from . import INDEXER_FIELDS, Config


def bf16_tensor(bits: np.ndarray, device="cpu"):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.to(device) if str(device) != "cpu" else t


def layer_config(w: synth.Workload, heads: int, T: Optional[int] = None, n_pos: Optional[int] = None,
                 t: Optional[int] = None, **kw) -> Config:
    base = dict(G=w.G, d_x=w.shape.d_x, H_I=w.shape.H_I)
    base.update(kw)
    return Config(H_kv=heads, T=w.T if T is None else T, n_pos=w.n_pos if n_pos is None else n_pos,
                  t=w.t if t is None else t, **base)


def layer_inputs_np(w: synth.Workload, layer: int, heads: Sequence[int], T: Optional[int] = None,
                    n_pos: Optional[int] = None, zero_value_path: bool = False) -> Dict[str, np.ndarray]:
    """bf16 bit arrays of one layer restricted to ``heads``:
    K, V [H][T][d]; Q [H][n][d]; X [n_pos][d_x]; indexer fields [H][...]."""
    pairs = [synth.make_pair(w, layer, h, T=T, n_pos=n_pos) for h in heads]
    idx = [synth.make_indexer(w, layer, h, zero_value_path=zero_value_path) for h in heads]
    out = {k: np.stack([p[k] for p in pairs]) for k in ("K", "V", "Q")}
    out["X"] = synth.make_layer_activations(w, layer, n_pos=n_pos)
    for f in INDEXER_FIELDS:
        out[f] = np.stack([ix[f] for ix in idx])
    return out


def to_device(arrs: Dict[str, np.ndarray], device="cuda", pin: bool = False):
    """bf16 bit arrays -> torch bf16 tensors (on ``device``, or pinned host memory)."""
    out = {}
    for k, v in arrs.items():
        t = bf16_tensor(v)
        if pin:
            out[k] = t.pin_memory()
        elif str(device) != "cpu":
            out[k] = t.to(device)
        else:
            out[k] = t
    return out


def indexer_dict(tens: Dict[str, object]) -> Dict[str, object]:
    return {f: tens[f] for f in INDEXER_FIELDS}
