"""C-ABI checks that need no GPU: the library loads, exports every function
declared in include/arckv.h, sizes workspaces, and rejects bad arguments on
the host before anything is enqueued."""
import re
from pathlib import Path

import pytest

import synth
import paper_2609_36835_gb300 as pk
from paper_2609_36835_gb300 import workload

HEADER = Path(__file__).resolve().parent.parent / "include" / "arckv.h"


def declared_functions():
    text = re.sub(r"/\*.*?\*/", "", HEADER.read_text(), flags=re.S)
    return sorted(set(re.findall(r"\b(arckv_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("arckv_compact", "arckv_attend", "arckv_workspace_bytes", "arckv_attend_workspace_bytes",
              "arckv_query_status", "arckv_status_string"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings(lib):
    for code in range(9):
        assert pk.status_string(code)
    assert pk.status_string(4) == "normal matrix of a fit is not positive definite"


def _cfg(**kw):
    w = synth.WORKLOADS["llama8b_layer_T8192"]
    return workload.layer_config(w, 8, **kw)


def test_workspace_bytes_sizes_and_rejections(lib):
    ws = pk.workspace_bytes(_cfg())
    # the n x T fp32 spill, its split-3 bf16 probabilities, k_bar and the t x t Gram dominate
    assert 0.8e9 < ws < 2.0e9
    assert pk.workspace_bytes(_cfg(t=9000)) == 0           # t > T
    assert pk.workspace_bytes(_cfg(t=0)) == 0
    assert pk.workspace_bytes(_cfg(d=64)) == 0             # unsupported head dim
    assert pk.workspace_bytes(_cfg(chunk_len=8192)) == 0   # chunked selection not built
    assert pk.attend_workspace_bytes(8, 1024, 819) > 0
    assert pk.attend_workspace_bytes(8, 1024, 0) == 0


@pytest.mark.parametrize("kw,code", [
    (dict(t=9000), 2), (dict(T=0), 2), (dict(H_I=17), 2), (dict(d_x=4095), 2), (dict(d=64), 8),
    (dict(chunk_len=4096), 8), (dict(lambda_m=1.5), 1), (dict(ridge_w=-1.0), 1), (dict(eps_w=0.0), 1),
    (dict(b_min=3.0, b_max=2.0), 1), (dict(flags=0x80), 1),
])
def test_compact_rejects_bad_config_without_gpu(lib, kw, code):
    idx = {f: 1 for f in pk.INDEXER_FIELDS}
    st, nl = pk.arckv_compact(_cfg(**kw), 1, 1, 1, 1, idx, 1, 1, 1, 256, 1 << 40, stream=0)
    assert st == code and nl == 0


def test_compact_rejects_null_pointers_and_small_workspace(lib):
    idx = {f: 1 for f in pk.INDEXER_FIELDS}
    cfg = _cfg()
    need = pk.workspace_bytes(cfg)
    assert pk.arckv_compact(cfg, None, 1, 1, 1, idx, 1, 1, 1, 256, need, stream=0)[0] == 1
    assert pk.arckv_compact(cfg, 1, 1, 1, 1, dict(idx, L_v=None), 1, 1, 1, 256, need, stream=0)[0] == 1
    assert pk.arckv_compact(cfg, 1, 1, 1, 1, idx, 1, 1, 1, 256, need - 1, stream=0)[0] == 3
    assert pk.arckv_compact(cfg, 1, 1, 1, 1, idx, 1, 1, 1, 258, need, stream=0)[0] == 3   # misaligned
    assert pk.arckv_compact(cfg, 1, 1, 1, 1, idx, 1, 1, 1, None, need, stream=0)[0] == 3
    # an assignment override needs an anchor override
    assert pk.arckv_compact(cfg, 1, 1, 1, 1, idx, 1, 1, 1, 256, need, stream=0, assign_in=8)[0] == 1


def test_attend_rejects_bad_arguments_without_gpu(lib):
    need = pk.attend_workspace_bytes(2, 16, 8)
    assert pk.arckv_attend(2, 16, 8, 64, 0.0, 1, 1, 1, 1, 1, 256, need, stream=0) == 8
    assert pk.arckv_attend(2, 16, 0, 128, 0.0, 1, 1, 1, 1, 1, 256, need, stream=0) == 2
    assert pk.arckv_attend(2, 16, 8, 128, 0.0, None, 1, 1, 1, 1, 256, need, stream=0) == 1
    assert pk.arckv_attend(2, 16, 8, 128, 0.0, 1, 1, 1, 1, 1, 256, need - 1, stream=0) == 3
    assert pk.arckv_attend(2, 16, 8, 128, -1.0, 1, 1, 1, 1, 1, 256, need, stream=0) == 1
    assert pk.arckv_attend(2, 16, 8, 128, 0.0, 1, 1, 1, 1, 1, 256, need, flags=4, stream=0) == 1
