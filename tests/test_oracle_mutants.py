"""Planted mistakes in the oracle must fail at least one of its pins.

Each case below is one plausible slip in ``oracle/arckv_oracle.py`` (a
dropped term, a wrong sign or index, a transposed or swapped operand, a
wrong tie rule).  The test plants it in a copy of the oracle's source text,
loads that copy as a module of its own, points the pin suite
(``tests/test_oracle_pins.py``) at it and runs the pins until one fails.  A
case that no pin catches means the pins leave that part of the oracle
unchecked.  The comparison helpers of ``oracle/parity.py`` get the same
treatment against ``tests/test_parity_helpers.py``.  Everything runs on the
CPU; the files on disk are not touched.
"""
import importlib.util
import sys
import types
from pathlib import Path

import numpy as np
import pytest

ROOT = Path(__file__).resolve().parent.parent
ORACLE_SRC = ROOT / "oracle" / "arckv_oracle.py"
PINS_SRC = Path(__file__).resolve().parent / "test_oracle_pins.py"
PARITY_SRC = ROOT / "oracle" / "parity.py"
PARITY_PINS_SRC = Path(__file__).resolve().parent / "test_parity_helpers.py"

# (name, exact fragment of the oracle's source, replacement)
MUTANTS = [
    # indexer, App. A.1
    ("param_count_drops_bias", "H_I * d_x + H_I + 3 * d_A", "H_I * d_x + 3 * d_A"),
    ("rms_norm_drops_1_over_dI", "keepdims=True) / d_I + 1e-6", "keepdims=True) + 1e-6"),
    ("value_context_keys_through_U_q", "(K @ U_k.T).T", "(K @ U_q.T).T"),
    ("value_context_keys_for_values", "c = A @ (V @ U_v.T)", "c = A @ (K @ U_v.T)"),
    ("projection_drops_value_context", "Q @ W[\"L_q\"].T + c @ W[\"L_c\"].T", "Q @ W[\"L_q\"].T"),
    ("projection_drops_value_key_path", "K @ W[\"L_k\"].T + V @ W[\"L_v\"].T", "K @ W[\"L_k\"].T"),
    ("key_blocks_not_normalised", "k_bar = rms_normalize(kz, d_I)", "k_bar = kz"),
    ("query_blocks_normalised_over_heads", "q_bar = rms_normalize(qz, d_I)",
     "q_bar = rms_normalize(qz.reshape(qz.shape[0], -1), d_I * qz.shape[1]).reshape(qz.shape)"),
    ("weights_drop_bias", "w = X_rows @ W[\"L_x\"].T + W[\"b_x\"][None, :]", "w = X_rows @ W[\"L_x\"].T"),
    ("leaky_slope_0_01", "x, 0.1 * x)", "x, 0.01 * x)"),
    ("leaky_sign_flipped", "np.where(x >= 0.0, x,", "np.where(x <= 0.0, x,"),
    ("index_drops_1_over_sqrt_dI", "k_bar[:, a, :].T) / np.sqrt(d_I)", "k_bar[:, a, :].T)"),
    ("index_weight_of_wrong_head", "I += w[:, a:a + 1] *", "I += w[:, 0:1] *"),
    ("pool_drops_square", "np.mean(pi * pi, axis=0)", "np.mean(pi, axis=0)"),
    ("pool_drops_root", "s = np.sqrt(np.mean(pi * pi, axis=0))", "s = np.mean(pi * pi, axis=0)"),
    # selection, Eq. persistent_support and App. A.3
    ("top_t_keeps_smallest", "np.lexsort((np.arange(s.shape[0]), -s))", "np.lexsort((np.arange(s.shape[0]), s))"),
    ("top_t_ties_to_higher_position", "np.lexsort((np.arange(s.shape[0]), -s))",
     "np.lexsort((-np.arange(s.shape[0]), -s))"),
    ("round_ties_to_odd", "(2 * r == den and q % 2 == 1)", "(2 * r == den and q % 2 == 0)"),
    ("round_ties_up", "(2 * r == den and q % 2 == 1)", "(2 * r == den)"),
    ("chunking_at_threshold", "if chunk_len <= 0 or T <= threshold:", "if chunk_len <= 0 or T < threshold:"),
    ("chunk_budget_floor_0", "min(max(round_half_even_ratio(t * Tc, T), 1), Tc)",
     "min(max(round_half_even_ratio(t * Tc, T), 0), Tc)"),
    ("chunk_budget_against_chunk_len", "round_half_even_ratio(t * Tc, T)", "round_half_even_ratio(t * Tc, chunk_len)"),
    ("chunked_positions_not_offset", "parts = [start + top_t(", "parts = [top_t("),
    # attention, profiles, assignment, merge (Sec. 3.4)
    ("logits_drop_scale", "return scale * (Q @ K.T)", "return Q @ K.T"),
    ("full_attention_keys_as_values", "return P, P @ V", "return P, P @ K"),
    ("profiles_normalised_over_rows", "return E / np.linalg.norm(E, axis=0, keepdims=True), M",
     "return E / np.linalg.norm(E, axis=1, keepdims=True), M"),
    ("profiles_not_normalised", "return E / np.linalg.norm(E, axis=0, keepdims=True), M", "return E, M"),
    ("assignment_argmin", "kappa[j0:j0 + rows] = np.argmax(sim, axis=1)",
     "kappa[j0:j0 + rows] = np.argmin(sim, axis=1)"),
    ("assignment_anchors_not_pinned", "    kappa[S] = np.arange(S.shape[0])\n", ""),
    ("mass_weights_drop_column_max", "return M + np.log(np.mean(", "return np.log(np.mean("),
    ("merge_lambda_swapped", "(1.0 - lambda_m) * K[S] + lambda_m * mu", "lambda_m * K[S] + (1.0 - lambda_m) * mu"),
    ("merge_weights_inverted", "wts = np.exp(logphi - gmax[kappa])", "wts = np.exp(gmax[kappa] - logphi)"),
    ("merge_unweighted_mean", "wts = np.exp(logphi - gmax[kappa])", "wts = np.ones_like(logphi)"),
    # fits (App. A.9)
    ("ridge_not_scaled_by_trace", "lam = ridge * np.trace(Gram) / t", "lam = ridge"),
    ("beta_global_shift", "    z = l.max(axis=1)\n    Phi_K", "    z = np.full(l.shape[0], l.max())\n    Phi_K"),
    ("beta_mass_over_columns", "m = Phi_K.sum(axis=1)", "m = Phi_K.mean(axis=1)"),
    ("beta_no_projection", "w_star = np.maximum(w_tilde, 0.0)", "w_star = np.abs(w_tilde)"),
    ("beta_no_clip", "beta = np.clip(np.log(np.maximum(w_star, cfg.eps_w)), cfg.b_min, cfg.b_max)",
     "beta = np.log(np.maximum(w_star, cfg.eps_w))"),
    ("values_beta_sign", "attention_logits(Q, C_k, scale) + beta[None, :])\n    _, Y",
     "attention_logits(Q, C_k, scale) - beta[None, :])\n    _, Y"),
    ("values_ridge_of_beta", "C_v = _ridge_solve(P_hat.T @ P_hat, P_hat.T @ Y, cfg.ridge_v)",
     "C_v = _ridge_solve(P_hat.T @ P_hat, P_hat.T @ Y, cfg.ridge_w)"),
    ("compact_attention_beta_dropped", "return _softmax_rows(attention_logits(Q, C_k, scale) + beta[None, :]) @ C_v",
     "return _softmax_rows(attention_logits(Q, C_k, scale)) @ C_v"),
    ("joint_bias_on_fixed_block", "b = np.concatenate([beta, np.zeros(K_fixed.shape[0])])",
     "b = np.concatenate([beta, np.ones(K_fixed.shape[0])])"),
    ("hard_subset_keys_as_values", "scale)) @ V[S]", "scale)) @ K[S]"),
    # HA / VI selectors and E(S), App. B.1
    ("ha_drops_square", "return np.sqrt(np.mean(P * P, axis=0))", "return np.sqrt(np.mean(P, axis=0))"),
    ("loo_p_instead_of_odds", "D = e / den * np.sqrt(dist2)", "D = e / msum * np.sqrt(dist2)"),
    ("loo_dominant_uses_full_output", "D[i, a[i]] = p_a * np.linalg.norm(V[a[i]] - O_minus)",
     "D[i, a[i]] = p_a * np.linalg.norm(V[a[i]] - O[i])"),
    ("vi_drops_square", "np.mean(D * D / (oo + eps), axis=0)", "np.mean(D / (oo + eps), axis=0)"),
    ("truncated_error_whole_norm", "/ (np.linalg.norm(O, axis=1) + eps)", "/ (np.linalg.norm(O) + eps)"),
    ("truncated_error_renormalised", "O_t = P[:, S] @ V[S]", "O_t = hard_subset_attention(Q_eval, K, V, S, scale)"),
    # diagnostics
    ("output_loss_unnormalised", "axis=1) / np.sum(y * y, axis=1))", "axis=1))"),
    ("mass_error_sign", "np.linalg.norm(Phi_C @ w_star - m)", "np.linalg.norm(Phi_C @ w_star + m)"),
    # axes and groupings
    ("projection_heads_grouped_wrongly", "qz = (Q @ W[\"L_q\"].T + c @ W[\"L_c\"].T).reshape(Q.shape[0], H_I, d_I)",
     "qz = (Q @ W[\"L_q\"].T + c @ W[\"L_c\"].T).reshape(Q.shape[0], d_I, H_I).transpose(0, 2, 1)"),
    ("value_context_softmax_over_queries", "    A = _softmax_rows(logits)\n", "    A = _softmax_rows(logits.T).T\n"),
    ("pool_softmax_over_queries", "    pi = _softmax_rows(I)\n", "    pi = _softmax_rows(I.T).T\n"),
    ("merge_not_normalised", "    mu = num / den[:, None]\n", "    mu = num\n"),
    ("loo_distance_sign", "dist2 = np.maximum(vv - 2.0 * (O @ V.T) + oo, 0.0)", "dist2 = np.maximum(vv + 2.0 * (O @ V.T) + oo, 0.0)"),
    ("pipeline_default_scale_1_over_d", "scale = cfg.scale if cfg.scale is not None else 1.0 / np.sqrt(d)",
     "scale = cfg.scale if cfg.scale is not None else 1.0 / d"),
    ("beta_fit_against_cache_keys", "Phi_C = np.exp(attention_logits(Q, C_k, scale) - z[:, None])",
     "Phi_C = np.exp(attention_logits(Q, C_k, 1.0) - z[:, None])"),
    # the pipeline of Sec. 3.2
    ("pipeline_merges_values", "C_k, _ = merge_keys(K, kappa, logphi, S, cfg.lambda_m)",
     "C_k, _ = merge_keys(V, kappa, logphi, S, cfg.lambda_m)"),
    ("pipeline_assignment_from_scores", "u, _ = response_profiles(l)", "u, _ = response_profiles(-l)"),
]


# slips in the comparison helpers the GPU parity tests rely on
PARITY_MUTANTS = [
    ("rel_fro_absolute", "return float(np.linalg.norm(a - b) / (nb if nb > 0 else 1.0))",
     "return float(np.linalg.norm(a - b))"),
    ("score_errors_top_t_only", "[: min(len(s), 2 * t)]", "[: min(len(s), t)]"),
    ("anchors_threshold_off_by_one", "k_thr = int(order[t - 1])", "k_thr = int(order[t])"),
    ("anchors_errors_narrow_the_band", "ok = all(g <= band + widen(j) for", "ok = all(g <= band - widen(j) for"),
    ("anchors_widening_uncapped", "return w if w <= WIDEN_CAP else 0.0", "return w"),
    ("anchors_widening_from_one_key", "w = err(j) + err(k_thr)", "w = err(j)"),
    ("anchors_errors_ignored", "return 0.0 if s_gpu is None else abs(float(s_gpu[j]) - s[j]) / abs(s[j])",
     "return 0.0"),
    ("anchors_no_size_check", "if len(a) != len(b) or len(S_gpu) != t:", "if False:"),
    ("chunked_scores_not_sliced", "s[start:start + Tc], tc, band, sg)", "s, tc, band, sg)"),
    ("chunked_positions_not_offset", "return X[(X >= start) & (X < start + Tc)] - start",
     "return X[(X >= start) & (X < start + Tc)]"),
    ("assignment_decided_rows_inverted", "    dec = (~is_anchor) & (gap > tau)\n    kappa_ref",
     "    dec = (~is_anchor) & (gap < tau)\n    kappa_ref"),
    ("assignment_anchor_rows_unchecked", "return (n_dec_mis == 0 and anchors_ok and worst <= tau)",
     "return (n_dec_mis == 0 and worst <= tau)"),
    ("assignment_shortfall_unchecked", "return (n_dec_mis == 0 and anchors_ok and worst <= tau)",
     "return (n_dec_mis == 0 and anchors_ok)"),
    ("profiles_form_wrong_block", "kg = kappa_gpu[j0:j0 + rows]", "kg = kappa_gpu[:rows][: sim.shape[0]]"),
    ("beta_support_everything", "sup = w_star > 1e-6 * wmax", "sup = w_star >= 0.0"),
    ("beta_rest_unchecked", "rest_ok = bool(np.all(beta_gpu[~sup] <= np.log(max(1e-5 * wmax, 1e-300)) + 1e-6))",
     "rest_ok = True"),
    ("mass_weights_in_log_space", "return rel_fro(np.exp(np.asarray(beta_gpu, dtype=np.float64)), "
     "np.exp(np.asarray(beta, dtype=np.float64)))", "return rel_fro(np.asarray(beta_gpu), np.asarray(beta))"),
]


# slips in the seeded input generator, against tests/test_synth_recipe.py
SYNTH_SRC = ROOT / "synth" / "__init__.py"
SYNTH_PINS_SRC = Path(__file__).resolve().parent / "test_synth_recipe.py"
SYNTH_MUTANTS = [
    ("outliers_x4", "k[:, _outlier_channels(w, layer)] *= 8.0", "k[:, _outlier_channels(w, layer)] *= 4.0"),
    ("no_attention_sink", "    k[0] *= 10.0\n", ""),
    ("device_no_attention_sink", "        k[0] = k[0] * 10.0\n", ""),
    ("device_rope_interleaved_pairs", "lo, hi = x[:, :half], x[:, half:]", "lo, hi = x[:, 0::2], x[:, 1::2]"),
    ("device_outliers_x4", "k[:, torch.as_tensor(_outlier_channels(w, layer), device=device)] *= 8.0",
     "k[:, torch.as_tensor(_outlier_channels(w, layer), device=device)] *= 4.0"),
    ("device_query_noise_1", "0.5 * torch.randn(n, D_HEAD", "1.0 * torch.randn(n, D_HEAD"),
    ("device_values_from_key_stream", "g.manual_seed(_torch_seed(w.wid, layer, h, _S_VALS))",
     "g.manual_seed(_torch_seed(w.wid, layer, h, _S_KEYS))"),
    ("rope_theta_10000", "ROPE_THETA = 500000.0", "ROPE_THETA = 10000.0"),
    ("rope_interleaved_pairs", "x1, x2 = x[:, :half], x[:, half:]", "x1, x2 = x[:, 0::2], x[:, 1::2]"),
    ("query_noise_1", "+ 0.5 * g.standard_normal((n, D_HEAD))", "+ 1.0 * g.standard_normal((n, D_HEAD))"),
    ("bf16_truncates", "u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16", "u = u >> 16"),
    ("bias_std_1", '"b_x": nrm((s.H_I,), 0.1)', '"b_x": nrm((s.H_I,), 1.0)'),
    ("outliers_reseeded_everywhere", "layer if w.outliers_per_layer else 0", "layer"),
    ("values_from_key_stream", "gv = _rng(w.wid, layer, head, _S_VALS)", "gv = _rng(w.wid, layer, head, _S_KEYS)"),
]


def _load(name: str, source: str, path: Path) -> types.ModuleType:
    mod = types.ModuleType(name)
    mod.__file__ = str(path)
    sys.modules[name] = mod   # dataclasses resolve their annotations through sys.modules
    try:
        exec(compile(source, str(path), "exec"), mod.__dict__)
    except BaseException:
        del sys.modules[name]
        raise
    return mod


def _run_pins(mod: types.ModuleType, stop_at_first: bool, pins_src: Path = PINS_SRC, attr: str = "oracle"):
    """Run every test of ``pins_src`` with its global ``attr`` bound to
    ``mod``.  Returns the names of the tests that raised."""
    spec = importlib.util.spec_from_file_location("_pins_under_mutation", pins_src)
    pins = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(pins)
    setattr(pins, attr, mod)
    failed = []
    for name in sorted(n for n in vars(pins) if n.startswith("test_")):
        fn = getattr(pins, name)
        if fn.__code__.co_argcount:   # parametrized tests need their arguments: not run here
            continue
        try:
            with np.errstate(all="ignore"):   # a slip may overflow; only the pin's verdict counts
                fn()
        except Exception:   # an AssertionError, or an error the slip provokes
            failed.append(name)
            if stop_at_first:
                break
    return failed


def _mutant_source(old: str, new: str, src_path: Path = ORACLE_SRC) -> str:
    src = src_path.read_text()
    assert src.count(old) == 1, f"fragment occurs {src.count(old)} times: {old!r}"
    return src.replace(old, new)


@pytest.mark.parametrize("src,pins,attr", [(ORACLE_SRC, PINS_SRC, "oracle"), (PARITY_SRC, PARITY_PINS_SRC, "parity"),
                                           (SYNTH_SRC, SYNTH_PINS_SRC, "synth")],
                         ids=["oracle", "parity", "synth"])
def test_unmodified_copy_passes_every_pin(src, pins, attr):
    mod = _load("_copy_" + attr, src.read_text(), src)
    try:
        assert _run_pins(mod, False, pins, attr) == []
    finally:
        del sys.modules["_copy_" + attr]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(name, old, new):
    mod_name = "_oracle_mutant_" + name
    mod = _load(mod_name, _mutant_source(old, new), ORACLE_SRC)
    try:
        assert _run_pins(mod, stop_at_first=True), f"no pin catches {name}"
    finally:
        del sys.modules[mod_name]


@pytest.mark.parametrize("name,old,new", PARITY_MUTANTS, ids=[m[0] for m in PARITY_MUTANTS])
def test_planted_mistake_in_parity_helpers_fails_a_check(name, old, new):
    mod_name = "_parity_mutant_" + name
    mod = _load(mod_name, _mutant_source(old, new, PARITY_SRC), PARITY_SRC)
    try:
        assert _run_pins(mod, True, PARITY_PINS_SRC, "parity"), f"no check catches {name}"
    finally:
        del sys.modules[mod_name]


@pytest.mark.parametrize("name,old,new", SYNTH_MUTANTS, ids=[m[0] for m in SYNTH_MUTANTS])
def test_planted_mistake_in_input_recipe_fails_a_check(name, old, new):
    mod_name = "_synth_mutant_" + name
    mod = _load(mod_name, _mutant_source(old, new, SYNTH_SRC), SYNTH_SRC)
    try:
        assert _run_pins(mod, True, SYNTH_PINS_SRC, "synth"), f"no check catches {name}"
    finally:
        del sys.modules[mod_name]
