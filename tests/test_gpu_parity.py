"""GPU-vs-oracle parity of arckv_compact / arckv_attend through the C ABI.

Tolerances are those stated in ``oracle/parity.py``.  Integer decisions
(anchors, assignment) are compared tie-aware.  The call a user makes (the
GPU's own anchors and assignment) is compared end to end: its compact
cache's attention output on held-out queries against the oracle's, and --
where its decisions equal the oracle's -- its C_k, beta and C_v.  The
floating-point outputs of the merge and the fits are also compared on the
oracle's own decisions, passed to the GPU through ``anchors_in`` /
``assign_in``.
"""
import os

import numpy as np
import pytest
import torch

import oracle
import synth
from oracle import parity
import paper_2609_36835_gb300 as pk
from paper_2609_36835_gb300 import workload

import conftest

pytestmark = pytest.mark.gpu

BAND = 1e-5   # relative score gap at the t-th score inside which anchors may trade places,
              # widened by the GPU scores' own errors at the two keys (parity.anchors_match)
TAU = 1e-4    # similarity gap inside which the assignment may differ (fp32 profile GEMM)


@pytest.fixture(scope="module", autouse=True)
def _gpu(lib):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def _ocfg(cfg: pk.Config):
    return oracle.OracleConfig(t=cfg.t, lambda_m=cfg.lambda_m, scale=(cfg.logit_scale or None),
                               ridge_w=cfg.ridge_w, ridge_v=cfg.ridge_v, eps_w=cfg.eps_w, b_min=cfg.b_min,
                               b_max=cfg.b_max, G=cfg.G, chunk_len=cfg.chunk_len,
                               selector={0: "indexer", 1: "ha", 2: "vi"}[cfg.selector])


def _pair64(arr, h, G):
    f64 = synth.bf16_to_f64
    K, V, Q = f64(arr["K"][h]), f64(arr["V"][h]), f64(arr["Q"][h])
    Xr = np.repeat(f64(arr["X"]), G, axis=0)
    W = {f: f64(arr[f][h]) for f in pk.INDEXER_FIELDS}
    return K, V, Q, Xr, W


def _run(cfg, ten, **kw):
    out = pk.compact_layer(cfg, ten["K"], ten["V"], ten["Q"], ten["X"], workload.indexer_dict(ten), **kw)
    torch.cuda.synchronize()
    return out


def _np(x):
    return x.detach().cpu().numpy()


def check_layer(w, heads, sample, T=None, n_pos=None, t=None, layer=0, n_hold=64, **cfgkw):
    """Full path on all ``heads``; oracle comparison on the ``sample`` heads."""
    arr = workload.layer_inputs_np(w, layer, heads, T=T, n_pos=n_pos)
    ten = workload.to_device(arr, "cuda")
    cfg = workload.layer_config(w, len(heads), T=T, n_pos=n_pos, t=t, **cfgkw)
    out = _run(cfg, ten, want_scores=True, want_assign=True)
    scale = cfg.logit_scale or 1.0 / np.sqrt(cfg.d)
    refs = {}
    for h in sample:
        K, V, Q, Xr, W = _pair64(arr, h, cfg.G)
        ref = oracle.compact_pair(K, V, Q, Xr, W, _ocfg(cfg), H_I=cfg.H_I)
        refs[h] = ref
        s_gpu = _np(out["scores"][h]).astype(np.float64)
        e_inf, e_top = parity.score_errors(s_gpu, ref["scores"], cfg.t)
        assert e_inf <= 1e-3 and e_top <= 1e-3, ("scores", h, e_inf, e_top)
        chunks = oracle.chunk_budgets(cfg.T, cfg.t, cfg.chunk_len)
        assert out["anchors"].shape[1] == len(ref["anchors"]) == sum(tc for _, _, tc in chunks)
        ok, nd, gap = parity.anchors_match_chunked(_np(out["anchors"][h]), ref["anchors"], ref["scores"], chunks, BAND,
                                                   s_gpu)
        assert ok, ("anchors", h, nd, gap)
        ref["_exch"], ref["_gap"] = nd, gap
    # downstream stages on the oracle's decisions (other heads keep the GPU's own)
    S_in = out["anchors"].clone()
    A_in = out["assign"].clone()
    for h in sample:
        S_in[h] = torch.as_tensor(refs[h]["anchors"], dtype=torch.int32)
        A_in[h] = torch.as_tensor(refs[h]["assign"], dtype=torch.int32)
    out2 = _run(cfg, ten, anchors_in=S_in, assign_in=A_in)
    out3 = _run(cfg, ten, anchors_in=S_in, want_assign=True)
    Qh = np.stack([synth.make_heldout(w, layer, h, arr["K"][i], n_hold) for i, h in enumerate(heads)])
    Qh_t = workload.bf16_tensor(Qh, "cuda")
    O = pk.attend(Qh_t, out2["C_k"], out2["beta"], out2["C_v"], cfg.logit_scale)
    O_user = pk.attend(Qh_t, out["C_k"], out["beta"], out["C_v"], cfg.logit_scale)
    for h in sample:
        ref = refs[h]
        # the call a user makes, end to end (Eq. compact_attention on held-out
        # queries).  Its decisions are integers taken at near-ties (anchor
        # scores within the tie band, assignment rows within TAU, some of them
        # 1e-13 apart); a tied row decided the other way moves its group's
        # merged key, and the fits and the held-out output with it, so the
        # end-to-end bound holds where the decisions agree, and the floating-
        # point stages are otherwise compared on the oracle's decisions below.
        O_ref = oracle.compact_attention(synth.bf16_to_f64(Qh[h]), ref["C_k"], ref["beta"], ref["C_v"], scale)
        e_user = parity.rel_fro(_np(O_user[h]), O_ref)
        same_S = np.array_equal(_np(out["anchors"][h]), ref["anchors"])
        n_ties = int(np.sum(_np(out["assign"][h]) != ref["assign"])) if same_S else -1
        compared = "decisions differ on tied keys"
        if same_S and n_ties == 0:
            # identical decisions: the unassisted outputs themselves
            assert e_user <= 2e-3, ("held-out output of the unassisted call", h, e_user)
            assert parity.rel_fro(_np(out["C_k"][h]), ref["C_k"]) <= 2e-3, ("unassisted C_k", h)
            eb, rest_ok = parity.beta_errors(_np(out["beta"][h]), ref["beta"], ref["w_star"])
            assert eb <= 2e-3 and rest_ok, ("unassisted beta", h, eb, rest_ok)
            assert parity.rel_fro(_np(out["C_v"][h]), ref["C_v"]) <= 2e-3, ("unassisted C_v", h)
            compared = "O,C_k,beta,C_v"
        elif same_S:
            # assignment differs on tied rows only (checked below): the merged
            # keys of the groups both sides formed alike must agree
            kg, kr = _np(out["assign"][h]), ref["assign"]
            moved = np.unique(np.concatenate([kg[kg != kr], kr[kg != kr]]))
            keep = np.setdiff1d(np.arange(len(ref["anchors"])), moved)
            assert parity.rel_fro(_np(out["C_k"][h])[keep], ref["C_k"][keep]) <= 2e-3, ("unassisted C_k rows", h)
            compared = "C_k(%d of %d groups)" % (len(keep), len(ref["anchors"]))
        conftest.PARITY_REPORT.append({
            "test": os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0].split("::")[-1], "head": h,
            "exch": ref.get("_exch", 0), "gap": ref.get("_gap", 0.0), "o_err": e_user,
            "ties": n_ties, "outputs": compared})
        assert parity.rel_fro(_np(out2["C_k"][h]), ref["C_k"]) <= 2e-3
        eb, rest_ok = parity.beta_errors(_np(out2["beta"][h]), ref["beta"], ref["w_star"])
        assert eb <= 2e-3 and rest_ok, ("beta", h, eb, rest_ok)
        assert parity.rel_fro(_np(out2["C_v"][h]), ref["C_v"]) <= 2e-3, ("C_v", h)
        assert parity.rel_fro(_np(O[h]), O_ref) <= 2e-3
        K, V, Q, Xr, W = _pair64(arr, h, cfg.G)
        u, _ = oracle.response_profiles(oracle.attention_logits(Q, K, scale))
        ok, n_mis, n_tie, worst = parity.assignment_valid_profiles(_np(out3["assign"][h]), u, ref["anchors"], TAU)
        assert ok, ("assign", h, n_mis, n_tie, worst)
    return cfg, arr, ten, out, out2


def test_small_single_head_workload():
    """T = 1024, one KV head, n = 256, t = 102 (the small workload in full)."""
    check_layer(synth.WORKLOADS["single_head_T1024"], [0], [0])


def test_ragged_tiles_two_heads():
    """T, n and t not multiples of the 128-wide tiles; two heads batched."""
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], [0, 3], [0, 1], T=1000, n_pos=50, t=77)


def test_full_llama_layer_sampled_heads():
    """One Llama-3.1-8B layer at full size (8 KV heads, T = 8192, n = 1024,
    t = 819) in the launch configuration the benchmark times; oracle on two heads."""
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], list(range(8)), [0, 7])


def test_many_row_tiles_single_k_split():
    """8 heads x 10 row tiles of reference rows (n = 1200): more row tiles than
    half the SMs, so the fused probability products run without a K split."""
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], list(range(8)), [3], T=2048, n_pos=300, t=205)


def test_many_reference_rows():
    """n = 2400 reference rows (n_pos = 600, GQA 4) against a short cache: the
    column statistics stage the longest row strips it supports."""
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], [4], [0], T=1024, n_pos=600, t=100)


def test_full_context_layer_retention_2pct():
    w = synth.WORKLOADS["llama8b_T8192_r02"]
    check_layer(w, list(range(8)), [5], layer=17)


def test_budget_above_reference_rows_uses_dual_fits():
    """t > n: the t x t normal matrices have rank <= n, the fits run in their
    n x n dual form (same ridge solution); compared with the primal oracle."""
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], [1, 6], [0, 1], T=1500, n_pos=40, t=300)


def test_full_context_layer_retention_5pct():
    """The 8K workload at 5% retention (t = 409) on a full layer of 8 heads."""
    check_layer(synth.WORKLOADS["llama8b_T8192_r05"], list(range(8)), [1, 6], layer=23)


# the sampled (layer, KV head) pairs on which the long-context workloads are
# checked against the oracle
LONG_PAIRS = [(0, 0), (15, 3), (31, 7)]


@pytest.mark.parametrize("layer,head", LONG_PAIRS, ids=["L%d_H%d" % p for p in LONG_PAIRS])
def test_long_context_32k_sampled_pairs(layer, head):
    """The 32K workload (T = 32768, n = 2048, t = 1638, outlier channels
    reseeded per layer) on one KV head per sampled pair."""
    check_layer(synth.WORKLOADS["llama8b_T32768_r05"], [head], [0], layer=layer, n_hold=32)


@pytest.mark.parametrize("layer,head", LONG_PAIRS, ids=["L%d_H%d" % p for p in LONG_PAIRS])
def test_long_context_128k_sampled_pairs(layer, head):
    """The 128K workload (T = 131072, n = 2048, t = 13107 > n, dual-form fits)
    on one KV head per sampled pair."""
    check_layer(synth.WORKLOADS["llama8b_T131072_r10"], [head], [0], layer=layer, n_hold=32)


def test_chunked_selection_32k_sampled_head():
    """App. A.3 chunked selection on the 32K workload: four 8192-chunks keep
    round(1638 / 4) = 410 anchors each (t' = 1640); merge and fits global."""
    cfg, *_ = check_layer(synth.WORKLOADS["llama8b_T32768_r05"], [4], [0], layer=3, n_hold=32, chunk_len=8192)
    assert pk.anchor_count(cfg) == 1640


def test_chunked_selection_ragged_last_chunk():
    """T = 20000 in chunks of 8192, 8192 and 3616 (budgets 819, 819, 362) on
    two heads, reference rows off the tile grid."""
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], [2, 5], [0, 1], T=20000, n_pos=60, t=2000, chunk_len=8192)


def test_chunked_selection_one_anchor_per_chunk():
    """Budgets clipped up to one anchor per chunk: T = 12000, chunks of 4096, t = 3."""
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], [1], [0], T=12000, n_pos=20, t=3, chunk_len=4096)


@pytest.mark.parametrize("selector", [pk.SELECTOR_HA, pk.SELECTOR_VI])
def test_ha_vi_selectors_small(selector):
    """App. B.1 selectors on the small workload, ragged shapes: scores, anchors
    (tie-aware) and the downstream stages on the oracle's anchors."""
    check_layer(synth.WORKLOADS["single_head_T1024"], [0], [0], selector=selector)
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], [1, 4], [0, 1], T=1000, n_pos=50, t=77, selector=selector)
    # T not a multiple of 4: the probability products take the unfused path
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], [3], [0], T=999, n_pos=30, t=50, selector=selector)


@pytest.mark.parametrize("selector", [pk.SELECTOR_HA, pk.SELECTOR_VI])
def test_ha_vi_selectors_full_layer_sampled_heads(selector):
    """HA / VI on a full Llama layer (8 heads, T = 8192, n = 1024, t = 819); oracle on two heads."""
    check_layer(synth.WORKLOADS["llama8b_layer_T8192"], list(range(8)), [2, 6], selector=selector)


def test_odd_shapes_single_index_head():
    """One index head, a narrow activation width and sizes off every tile."""
    w = synth.Workload("odd_shapes", 11, 1, 2, 333, 7, 5, shape=synth.IndexerShape(H_I=1, d_x=72))
    check_layer(w, [0, 1], [1])


@pytest.mark.parametrize("t", [1, 2])
def test_tiny_budgets(t):
    check_layer(synth.WORKLOADS["single_head_T1024"], [0], [0], T=200, n_pos=16, t=t)


@pytest.mark.parametrize("lam", [0.0, 1.0])
def test_merge_endpoints(lam):
    w = synth.WORKLOADS["single_head_T1024"]
    cfg, arr, ten, out, out2 = check_layer(w, [0], [0], T=500, n_pos=32, t=40, lambda_m=lam)
    if lam == 0.0:   # C_k = K_S exactly
        K = synth.bf16_to_f32(arr["K"][0])
        S = _np(out["anchors"][0])
        assert np.array_equal(_np(_run(cfg, ten)["C_k"][0]), K[S])


def test_identity_budget_reproduces_cache():
    """t = T: every group is a singleton, so C_k = K bit for bit.  With the
    keys themselves as reference queries (Gaussian keys, no attention sink)
    Phi_C is near the identity and the unregularised fits are well
    conditioned, so beta = 0 and C_v = V up to fp32 rounding."""
    w = synth.WORKLOADS["single_head_T1024"]
    arr = workload.layer_inputs_np(w, 0, [0], T=64, n_pos=16)
    rng = np.random.default_rng(5)
    arr["K"] = synth.bf16_round(rng.normal(size=(1, 64, 128)).astype(np.float32))
    arr["V"] = synth.bf16_round(rng.normal(size=(1, 64, 128)).astype(np.float32))
    arr["Q"] = arr["K"].copy()
    ten = workload.to_device(arr, "cuda")
    cfg = workload.layer_config(w, 1, T=64, n_pos=16, t=64, ridge_w=0.0, ridge_v=0.0, lambda_m=0.6)
    out = _run(cfg, ten)
    K = synth.bf16_to_f32(arr["K"][0])
    assert np.array_equal(_np(out["anchors"][0]), np.arange(64))
    assert np.array_equal(_np(out["C_k"][0]), K)
    assert np.max(np.abs(_np(out["beta"][0]))) <= 1e-5
    assert parity.rel_fro(_np(out["C_v"][0]), synth.bf16_to_f32(arr["V"][0])) <= 1e-5


@pytest.mark.parametrize("T,n_pos", [(2048, 64), (20000, 60)])
def test_bitwise_reproducible(T, n_pos):
    """Two calls give identical bits; T = 20000 ends in a 32-column tile, so
    the staged logit stores skip boxes past the last column."""
    w = synth.WORKLOADS["llama8b_layer_T8192"]
    arr = workload.layer_inputs_np(w, 1, [0, 1], T=T, n_pos=n_pos)
    ten = workload.to_device(arr, "cuda")
    cfg = workload.layer_config(w, 2, T=T, n_pos=n_pos, t=T // 10)
    a = _run(cfg, ten, want_scores=True, want_assign=True)
    for _ in range(3):
        b = _run(cfg, ten, want_scores=True, want_assign=True)
        for k in ("scores", "anchors", "assign", "C_k", "beta", "C_v"):
            assert torch.equal(a[k], b[k]), k


def test_nonblocking_then_query_status():
    w = synth.WORKLOADS["single_head_T1024"]
    arr = workload.layer_inputs_np(w, 0, [0], T=256, n_pos=16)
    ten = workload.to_device(arr, "cuda")
    cfg = workload.layer_config(w, 1, T=256, n_pos=16, t=20, flags=pk.FLAG_NONBLOCKING)
    ws = torch.empty(pk.workspace_bytes(cfg), dtype=torch.uint8, device="cuda")
    out = _run(cfg, ten, ws=ws)
    assert out["status"] == 0
    assert pk.arckv_query_status(ws) == 0
    blocking = workload.layer_config(w, 1, T=256, n_pos=16, t=20)
    ref = _run(blocking, ten)
    assert torch.equal(out["C_v"], ref["C_v"])


def test_bounded_wait_gives_up_and_context_stays_usable():
    """Failure detection without a GPU fault: a bounded device wait on an
    mbarrier that nothing completes gives up after 20 ms and reports
    ARCKV_ERR_TIMEOUT through the status word; the next compaction on the same
    context runs normally."""
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    assert pk.arckv_wait_probe(ws, 256, 20000) == 6
    assert pk.arckv_query_status(ws) == 6   # still recorded; reading it clears it
    assert pk.arckv_query_status(ws) == 0
    w = synth.WORKLOADS["single_head_T1024"]
    arr = workload.layer_inputs_np(w, 0, [0], T=256, n_pos=16)
    cfg = workload.layer_config(w, 1, T=256, n_pos=16, t=20)
    out = _run(cfg, workload.to_device(arr, "cuda"))
    assert out["status"] == 0 and bool(torch.isfinite(out["C_v"]).all())


def test_nonfinite_input_is_reported():
    w = synth.WORKLOADS["single_head_T1024"]
    arr = workload.layer_inputs_np(w, 0, [0], T=256, n_pos=16)
    ten = workload.to_device(arr, "cuda")
    ten["K"][0, 17, 3] = float("nan")
    cfg = workload.layer_config(w, 1, T=256, n_pos=16, t=20)
    out = _run(cfg, ten, check=False)
    assert out["status"] == 5
    # the context stays usable
    ten2 = workload.to_device(arr, "cuda")
    assert _run(cfg, ten2)["status"] == 0


def test_singular_fit_returns_not_spd():
    """Q = 0 makes every logit 0 and Phi_C the all-ones matrix, whose Gram
    n 11^T is singular for t >= 2; with ridge_w = 0 the factorisation meets an
    exactly zero pivot and the call returns ARCKV_ERR_NOT_SPD."""
    w = synth.WORKLOADS["single_head_T1024"]
    arr = workload.layer_inputs_np(w, 0, [0], T=128, n_pos=64)
    ten = workload.to_device(arr, "cuda")
    ten["Q"].zero_()
    cfg = workload.layer_config(w, 1, T=128, n_pos=64, t=4, ridge_w=0.0)
    S = torch.tensor([[0, 1, 2, 3]], dtype=torch.int32, device="cuda")
    out = _run(cfg, ten, anchors_in=S, check=False)
    assert out["status"] == 4
    assert _run(workload.layer_config(w, 1, T=128, n_pos=64, t=4), workload.to_device(arr, "cuda"))["status"] == 0


def test_invalid_overrides_are_rejected_on_device():
    w = synth.WORKLOADS["single_head_T1024"]
    arr = workload.layer_inputs_np(w, 0, [0], T=128, n_pos=8)
    ten = workload.to_device(arr, "cuda")
    cfg = workload.layer_config(w, 1, T=128, n_pos=8, t=4)
    bad = torch.tensor([[5, 3, 9, 400]], dtype=torch.int32, device="cuda")
    assert _run(cfg, ten, anchors_in=bad, check=False)["status"] == 1
    S = torch.tensor([[1, 5, 9, 100]], dtype=torch.int32, device="cuda")
    A = torch.full((1, 128), 7, dtype=torch.int32, device="cuda")
    assert _run(cfg, ten, anchors_in=S, assign_in=A, check=False)["status"] == 1
    assert _run(cfg, ten)["status"] == 0


@pytest.mark.parametrize("H,n,t", [(3, 200, 77), (1, 1, 1), (2, 130, 300)])
def test_attend_matches_oracle(H, n, t):
    rng = np.random.default_rng(H * 1000 + t)
    Qb = synth.bf16_round((rng.normal(size=(H, n, 128)) * 3).astype(np.float32))
    Ck = rng.normal(size=(H, t, 128)).astype(np.float32)
    beta = rng.normal(size=(H, t)).astype(np.float32)
    Cv = rng.normal(size=(H, t, 128)).astype(np.float32)
    O = pk.attend(workload.bf16_tensor(Qb, "cuda"), torch.from_numpy(Ck).cuda(), torch.from_numpy(beta).cuda(),
                  torch.from_numpy(Cv).cuda())
    for h in range(H):
        ref = oracle.compact_attention(synth.bf16_to_f64(Qb[h]), Ck[h].astype(np.float64),
                                       beta[h].astype(np.float64), Cv[h].astype(np.float64), 1.0 / np.sqrt(128))
        assert parity.rel_fro(_np(O[h]), ref) <= 2e-3
