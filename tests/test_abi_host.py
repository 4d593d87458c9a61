"""C-ABI checks that need no GPU: the library loads, exports every function
declared in include/arckv.h, sizes workspaces, and rejects bad arguments on
the host before anything is enqueued."""
import re
from pathlib import Path

import numpy as np
import pytest

import oracle
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
              "arckv_query_status", "arckv_status_string", "arckv_anchor_count", "arckv_attend_joint",
              "arckv_attend_joint_workspace_bytes"):
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
    return workload.layer_config(w, kw.pop("H_kv", 8), **kw)


def test_workspace_bytes_sizes_and_rejections(lib):
    ws = pk.workspace_bytes(_cfg())
    # the n x T fp32 spill, k_bar, the transposed profiles and the t x t Gram dominate
    assert 0.8e9 < ws < 2.0e9
    assert pk.workspace_bytes(_cfg(t=9000)) == 0           # t > T
    assert pk.workspace_bytes(_cfg(t=0)) == 0
    assert pk.workspace_bytes(_cfg(d=64)) == 0             # unsupported head dim
    assert pk.workspace_bytes(_cfg(chunk_len=4096)) == ws  # T = 8192 <= 10,000: chunking is bypassed
    assert pk.attend_workspace_bytes(8, 1024, 819) > 0
    assert pk.attend_workspace_bytes(8, 1024, 0) == 0


def test_long_context_workspaces_fit_the_bench(lib):
    """The dual-form workspace of a 128K layer call (8 heads) and the 32K one:
    the bench holds three 128K workspaces beside a 17.8 GB context in HBM."""
    w128 = synth.WORKLOADS["llama8b_T131072_r10"]
    ws128 = pk.workspace_bytes(workload.layer_config(w128, w128.H_kv))
    assert 20e9 < ws128 < 30e9
    w32 = synth.WORKLOADS["llama8b_T32768_r05"]
    ws32 = pk.workspace_bytes(workload.layer_config(w32, w32.H_kv))
    assert 4e9 < ws32 < 8e9
    assert 3 * ws128 + 17.8e9 < 200e9


def test_wait_probe_rejects_bad_arguments_on_the_host(lib):
    assert pk.arckv_wait_probe(None, 256, 1000, stream=0) == 3     # no workspace
    assert pk.arckv_wait_probe(None, 256, 0, stream=0) == 1        # limit out of range
    assert pk.arckv_wait_probe(None, 256, 2000000, stream=0) == 1


def test_probability_triple_only_when_t_not_tileable(lib):
    """softmax(X) V runs fused (no probability triple in the workspace) when T
    is a multiple of 4; one key more and the unfused path's three bf16 n x T
    arrays are allocated."""
    cfg = _cfg(T=8192)
    H, n = cfg.H_kv, cfg.n_pos * cfg.G
    extra = pk.workspace_bytes(_cfg(T=8193)) - pk.workspace_bytes(cfg)
    triple = 3 * H * n * 8200 * 2   # three bf16 arrays with rows padded to a multiple of 8
    assert triple <= extra < triple + 64 * 1024 * 1024


@pytest.mark.parametrize("kw,code", [
    (dict(t=9000), 2), (dict(T=0), 2), (dict(H_I=17), 2), (dict(d_x=4095), 2), (dict(d=64), 8),
    (dict(chunk_len=-1), 1), (dict(T=1 << 20, chunk_len=8), 2), (dict(selector=3), 1), (dict(selector=-1), 1),
    (dict(selector=2, T=1, t=1), 2), (dict(lambda_m=1.5), 1), (dict(ridge_w=-1.0), 1), (dict(eps_w=0.0), 1),
    (dict(b_min=3.0, b_max=2.0), 1), (dict(flags=0x80), 1),
    (dict(logit_scale=float("nan")), 1), (dict(logit_scale=float("inf")), 1), (dict(lambda_m=float("nan")), 1),
    (dict(ridge_v=float("inf")), 1), (dict(b_max=float("inf")), 1), (dict(eps_w=float("nan")), 1),
    (dict(n_pos=65536), 2),            # n T = 2^31: per-head offsets would leave 32 bits
    (dict(H_kv=8192), 2),              # H_kv times the K slices exceeds the grid's y limit
    (dict(t=50000, T=60000), 2),       # t^2 >= 2^31
])
def test_compact_rejects_bad_config_without_gpu(lib, kw, code):
    idx = {f: 1 for f in pk.INDEXER_FIELDS}
    st, nl = pk.arckv_compact(_cfg(**kw), 1, 1, 1, 1, idx, 1, 1, 1, 256, 1 << 40, stream=0)
    assert st == code and nl == 0


def test_anchor_count_matches_the_oracle_budgets(lib):
    """Realized anchors per head (App. A.3), integer-exact against the oracle."""
    w32 = synth.WORKLOADS["llama8b_T32768_r05"]
    assert pk.anchor_count(workload.layer_config(w32, 8, chunk_len=8192)) == 1640
    assert pk.anchor_count(workload.layer_config(w32, 8)) == 1638
    w128 = synth.WORKLOADS["llama8b_T131072_r10"]
    assert pk.anchor_count(workload.layer_config(w128, 8, chunk_len=8192)) == 13104
    assert pk.anchor_count(_cfg(chunk_len=4096)) == 819          # bypassed at T = 8192
    assert pk.anchor_count(_cfg(t=0)) == 0
    rng = np.random.default_rng(0)
    for _ in range(200):
        T = int(rng.integers(10001, 200000))
        L = int(rng.integers(512, 40000))
        t = int(rng.integers(1, min(T // 4, 30000)))   # t^2 < 2^31 keeps the config valid
        assert pk.anchor_count(_cfg(T=T, t=t, chunk_len=L)) == oracle.anchor_count(T, t, L), (T, t, L)
    # exact halves go to the even neighbour
    assert pk.anchor_count(_cfg(T=20000, t=5, chunk_len=10000)) == 4
    assert pk.anchor_count(_cfg(T=20000, t=7, chunk_len=10000)) == 8
    ws_c = pk.workspace_bytes(workload.layer_config(w32, 8, chunk_len=8192))
    ws_g = pk.workspace_bytes(workload.layer_config(w32, 8))
    assert ws_c > ws_g > 0   # two more anchors per head


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


def test_attend_joint_rejects_bad_arguments_without_gpu(lib):
    need = pk.attend_joint_workspace_bytes(2, 4, 8, 8)
    assert need > 0
    args = dict(H=2, n=4, t=8, F=8, d=128, logit_scale=0.0, Q=256, C_k=256, beta=256, C_v=256, K_fixed=256,
                V_fixed=256, O=256, ws=256, ws_bytes=need, stream=0)
    call = lambda **kw: pk.arckv_attend_joint(**dict(args, **kw))
    assert call(d=64) == 8
    assert call(t=0, F=0) == 2
    assert call(C_k=None) == 1
    assert call(K_fixed=None) == 1
    assert call(C_v=264) == 1            # not 16-byte aligned
    assert call(ws_bytes=need - 1) == 3
    assert call(flags=0x4) == 1
    assert call(logit_scale=-1.0) == 1


def test_torch_helpers_validate_arguments_before_the_library():
    """Wrong dtype, shape or layout, or host tensors, are refused by the
    binding itself: nothing reaches the library, and there is no CPU path."""
    import torch
    cfg = _cfg(T=64, n_pos=4, t=8, H_kv=2)
    bf = lambda *s: torch.zeros(*s, dtype=torch.bfloat16)
    K = bf(2, 64, 128)
    with pytest.raises(ValueError, match="contiguous"):
        pk._ptr(torch.zeros(4, 4).t())
    with pytest.raises(ValueError, match="K must be torch.bfloat16"):
        pk.compact_layer(cfg, K.float(), K, bf(2, 16, 128), bf(4, cfg.d_x), {})
    with pytest.raises(ValueError, match="K must have shape"):
        pk.compact_layer(cfg, bf(2, 65, 128), K, bf(2, 16, 128), bf(4, cfg.d_x), {})
    with pytest.raises(ValueError, match="indexer.L_q must be a torch tensor"):
        pk.compact_layer(cfg, K, K, bf(2, 16, 128), bf(4, cfg.d_x), {})
    with pytest.raises(ValueError, match="anchors_in must have shape"):
        pk.compact_layer(cfg, K, K, bf(2, 16, 128), None, None, anchors_in=torch.zeros(2, 7, dtype=torch.int32))
    with pytest.raises(ValueError, match="K must be on a CUDA device"):
        pk.compact_layer(cfg, K, K, bf(2, 16, 128), None, None, anchors_in=torch.zeros(2, 8, dtype=torch.int32))
    f32 = lambda *s: torch.zeros(*s, dtype=torch.float32)
    with pytest.raises(ValueError, match="beta must be torch.float32"):
        pk.attend(bf(2, 4, 128), f32(2, 8, 128), torch.zeros(2, 8, dtype=torch.float64), f32(2, 8, 128))
    with pytest.raises(ValueError, match="CUDA device"):
        pk.attend(bf(2, 4, 128), f32(2, 8, 128), f32(2, 8), f32(2, 8, 128))
    with pytest.raises(ValueError, match="together"):
        pk.attend_joint(bf(2, 4, 128), f32(2, 8, 128), f32(2, 8), None)
    with pytest.raises(ValueError, match="C_v must be torch.float32"):
        pk.attend_joint(bf(2, 4, 128), f32(2, 8, 128), f32(2, 8), bf(2, 8, 128))
    with pytest.raises(ValueError, match="S must be torch.int32"):
        pk.truncated_error(bf(2, 4, 128), K, K, torch.zeros(2, 8, dtype=torch.int64))


def test_plain_c_program_uses_the_header_and_library(lib, tmp_path):
    """The boundary is a C ABI: a C99 program (tests/abi_consumer.c) compiles
    against include/arckv.h with -pedantic, links libarckv.so, and gets the
    same host-side answers as the Python binding."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    root = Path(__file__).resolve().parent.parent
    pkg = root / "paper_2609_36835_gb300"
    exe = tmp_path / "abi_consumer"
    subprocess.run([gcc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", str(root / "include"),
                    str(root / "tests" / "abi_consumer.c"), "-L", str(pkg), "-larckv", "-Wl,-rpath," + str(pkg),
                    "-o", str(exe)], check=True)
    out = dict(l.split(" ", 1) for l in subprocess.run([str(exe)], check=True, capture_output=True,
                                                         text=True).stdout.splitlines())
    assert int(out["workspace_bytes"]) == pk.workspace_bytes(_cfg()) > 0
    assert int(out["workspace_bytes_bad"]) == 0
    w32 = synth.WORKLOADS["llama8b_T32768_r05"]
    assert int(out["anchor_count_chunked"]) == pk.anchor_count(workload.layer_config(w32, 8, chunk_len=8192)) == 1640
    assert int(out["attend_workspace_bytes"]) == pk.attend_workspace_bytes(2, 16, 8)
    for code in range(9):
        assert out["status_%d" % code] == pk.status_string(code)
    assert int(out["compact_null_config"]) == 1 and int(out["compact_bad_shape"]) == 2
