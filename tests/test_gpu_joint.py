"""GPU-vs-oracle parity of arckv_attend_joint (App. A.7 joint attention with
an uncompressed block) through the C ABI.

The kernel reads exact inputs (bf16 queries and caches, fp32 or bf16 compact
rows) and accumulates in fp32 with an fp32 softmax; its error is a few fp32
roundings per key weight, so outputs are held to a relative Frobenius error
of 1e-4 against the fp64 oracle (tighter than the 2e-3 of the fitted outputs).
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from oracle import parity
import paper_2609_36835_gb300 as pk
from paper_2609_36835_gb300 import workload

pytestmark = pytest.mark.gpu
TOL = 1e-4
SC = 1.0 / np.sqrt(128.0)


@pytest.fixture(scope="module", autouse=True)
def _gpu(lib):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def _case(heads, T, t, F, n, layer=0, compact_bf16=False):
    """Per head: fixed block = the last F rows of a Llama-shaped pair's cache,
    compact block = a stand-in compact cache drawn from its first T - F rows."""
    w = synth.WORKLOADS["llama8b_layer_T8192"]
    host = []
    for h in heads:
        p = synth.make_pair(w, layer, h, T=T, n_pos=max(1, (n + w.G - 1) // w.G))
        cc = synth.make_compact_cache(w, layer, h, p["K"][:T - F], p["V"][:T - F], t)
        if compact_bf16:
            cc = {k: (synth.bf16_round(v) if k != "beta" else v) for k, v in cc.items()}
        host.append(dict(Q=p["Q"][:n], Kf=p["K"][T - F:], Vf=p["V"][T - F:], **cc))
    return host


def _run(host, compact_bf16=False, with_compact=True, with_fixed=True):
    def bf(key):
        return workload.bf16_tensor(np.stack([x[key] for x in host]), "cuda")
    def ck(key):
        a = np.stack([x[key] for x in host])
        if compact_bf16 and key != "beta":
            return workload.bf16_tensor(a, "cuda")
        return torch.as_tensor(a, device="cuda")
    O = pk.attend_joint(bf("Q"), ck("C_k") if with_compact else None, ck("beta") if with_compact else None,
                        ck("C_v") if with_compact else None, bf("Kf") if with_fixed else None,
                        bf("Vf") if with_fixed else None)
    torch.cuda.synchronize()
    return O.cpu().numpy()


def _ref(x, compact_bf16=False, with_compact=True, with_fixed=True):
    f64 = synth.bf16_to_f64
    Q = f64(x["Q"])
    if with_compact:
        C_k = f64(x["C_k"]) if compact_bf16 else x["C_k"].astype(np.float64)
        C_v = f64(x["C_v"]) if compact_bf16 else x["C_v"].astype(np.float64)
        beta = x["beta"].astype(np.float64)
    else:
        C_k = C_v = np.zeros((0, 128))
        beta = np.zeros(0)
    Kf, Vf = (f64(x["Kf"]), f64(x["Vf"])) if with_fixed else (np.zeros((0, 128)), np.zeros((0, 128)))
    return oracle.joint_compact_attention(Q, C_k, beta, C_v, Kf, Vf, SC)


@pytest.mark.parametrize("compact_bf16", [False, True])
def test_joint_ragged_rows_and_straddling_tiles(compact_bf16):
    """n = 5 rows, t = 77 compact and F = 130 uncompressed keys: tiles cross
    the block boundary and row blocks are partial."""
    host = _case([0, 3, 6], T=1200, t=77, F=130, n=5, compact_bf16=compact_bf16)
    O = _run(host, compact_bf16)
    for i, x in enumerate(host):
        assert parity.rel_fro(O[i], _ref(x, compact_bf16)) <= TOL


def test_joint_fixed_block_only_is_plain_attention():
    host = _case([1, 2], T=3000, t=10, F=2500, n=4)
    O = _run(host, with_compact=False)
    for i, x in enumerate(host):
        _, O_full = oracle.full_attention(synth.bf16_to_f64(x["Q"]), synth.bf16_to_f64(x["Kf"]),
                                          synth.bf16_to_f64(x["Vf"]), SC)
        assert parity.rel_fro(O[i], O_full) <= TOL


def test_joint_compact_block_only_matches_oracle_and_arckv_attend():
    host = _case([4, 5], T=2000, t=409, F=1, n=64)
    O = _run(host, with_fixed=False)
    Q = workload.bf16_tensor(np.stack([x["Q"] for x in host]), "cuda")
    ck = {k: torch.as_tensor(np.stack([x[k] for x in host]), device="cuda") for k in ("C_k", "beta", "C_v")}
    O2 = pk.attend(Q, ck["C_k"], ck["beta"], ck["C_v"]).cpu().numpy()
    for i, x in enumerate(host):
        r = _ref(x, with_fixed=False)
        assert parity.rel_fro(O[i], r) <= TOL
        assert parity.rel_fro(O2[i], r) <= TOL


def test_joint_long_key_range_many_splits():
    """40,000 keys in one head: many key splits merged by the combine pass."""
    host = _case([7], T=40000, t=3000, F=30000, n=4)
    O = _run(host)
    assert parity.rel_fro(O[0], _ref(host[0])) <= TOL


def test_joint_single_key():
    host = _case([0], T=64, t=1, F=0, n=2)
    O = _run(host, with_fixed=False)
    # one key: the output is its value row exactly (softmax weight 1)
    assert np.allclose(O[0], np.broadcast_to(host[0]["C_v"][0], (2, 128)), rtol=0, atol=1e-6)


def test_decode_batch_full_size_sampled_heads():
    """The decode configuration the benchmark times: batch 64 x 8 KV heads
    (H = 512), G = 4 rows each, T = 8192 full cache vs the t = 1638 (20 %)
    bf16 compact cache with an F = 0 fixed block; oracle on sampled heads."""
    H, G, T, t = 512, 4, 8192, 1638
    d = synth.decode_batch_device(11, H, G, T, t, 0, "cuda", compact_bf16=True)
    O_full = pk.attend_joint(d["Q"], K_fixed=d["K"], V_fixed=d["V"])
    O_comp = pk.attend_joint(d["Q"], d["C_k"], d["beta"], d["C_v"])
    torch.cuda.synchronize()
    for h in (0, 137, 511):
        f = lambda x: x[h].float().cpu().double().numpy()
        Q = f(d["Q"])
        _, ref_full = oracle.full_attention(Q, f(d["K"]), f(d["V"]), SC)
        assert parity.rel_fro(O_full[h].cpu().numpy(), ref_full) <= TOL
        ref_c = oracle.compact_attention(Q, f(d["C_k"]), f(d["beta"]), f(d["C_v"]), SC)
        assert parity.rel_fro(O_comp[h].cpu().numpy(), ref_c) <= TOL


@pytest.mark.parametrize("layer_heads,T,n_pos,t", [((0, [0, 3]), 1000, 50, 77), ((2, list(range(8))), 8192, 256, 819)])
def test_truncated_output_error_of_the_three_selectors(layer_heads, T, n_pos, t):
    """E(S) (App. B.1) on held-out queries for the anchor sets of the indexer,
    HA and VI selectors, against the oracle (relative 1e-4)."""
    layer, heads = layer_heads
    w = synth.WORKLOADS["llama8b_layer_T8192"]
    arr = workload.layer_inputs_np(w, layer, heads, T=T, n_pos=n_pos)
    ten = workload.to_device(arr, "cuda")
    Qh = np.stack([synth.make_heldout(w, layer, h, arr["K"][i], 64) for i, h in enumerate(heads)])
    Qt = workload.bf16_tensor(Qh, "cuda")
    results = {}
    for sel in (pk.SELECTOR_INDEXER, pk.SELECTOR_HA, pk.SELECTOR_VI):
        cfg = workload.layer_config(w, len(heads), T=T, n_pos=n_pos, t=t, selector=sel)
        out = pk.compact_layer(cfg, ten["K"], ten["V"], ten["Q"], ten["X"], workload.indexer_dict(ten))
        E = pk.truncated_error(Qt, ten["K"], ten["V"], out["anchors"]).cpu().numpy()
        S = out["anchors"].cpu().numpy()
        for i in (0, len(heads) - 1):
            ref = oracle.truncated_output_error(synth.bf16_to_f64(Qh[i]), synth.bf16_to_f64(arr["K"][i]),
                                                synth.bf16_to_f64(arr["V"][i]), S[i], SC)
            assert abs(E[i] - ref) <= 1e-4 * ref, (sel, i, E[i], ref)
        results[sel] = E
    # empty and full sets: E = mean ||O|| / (||O|| + eps) ~ 1 and E = 0
    Sall = torch.arange(T, dtype=torch.int32, device="cuda").repeat(len(heads), 1)
    assert np.all(pk.truncated_error(Qt, ten["K"], ten["V"], Sall).cpu().numpy() < 1e-5)
    E0 = pk.truncated_error(Qt, ten["K"], ten["V"], None).cpu().numpy()
    assert np.allclose(E0, 1.0, atol=1e-5)
