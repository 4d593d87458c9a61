"""fp64 CPU oracle for ARC-KV per-context KV-cache compaction.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline / reference legs of ``bench.py`` may import this module.
It shares no code with the CUDA library (``paper_2609_36835_gb300``) and
never imports it; the two meet only in the seeded input generator
``synth``, which holds none of the method's arithmetic.

Every function below states one definition of the paper, evaluated in
float64 from the exact (bf16-widened) inputs, in the paper's order and
notation, for ONE layer-KV-head pair.  Matrix products, softmax maxima and
the Cholesky factorisation are library primitives (numpy / scipy); there is
no blocking, fusion or reformulation beyond what the cited equation states.

Notation: T cache rows, d head dim, n reference-query rows of this KV head
(row i = r*G + g pairs reference position r with query head g), t budget.

Readings of points the paper leaves open:

* ``scale``: the paper omits the 1/sqrt(d) factor of attention logits as a
  notational convention (Sec. 3.1).  Every model-attention logit q.k here is
  multiplied by ``scale`` (default 1/sqrt(d)); the indexer's own logits are
  used exactly as printed (value head unscaled, index head divided by
  sqrt(d_I)), App. A.1.
* top-t ties go to the lower position; S is returned in ascending order.
* assignment ties go to the smallest anchor index r (App. A.8 leaves the
  tie rule open beyond being deterministic).
* both least-squares fits are solved with a ridge lam = ridge * tr(Gram)/t;
  ridge = 0 is the paper's unregularised solve for beta (Eq. mass_fit).
* eps_w, b_min, b_max (unstated in Eq. mass_fit) default to e^-20, -20, 20.
* the epsilon of the HA/VI selectors and of E(S) (App. B.1, unstated) is 1e-6;
  the leave-one-out change of a row's dominant column is evaluated in its
  exact algebraic form p_a ||v_a - O^(-a)|| (see leave_one_out_changes).
* chunked selection (App. A.3, ``chunk_len`` > 0, T above 10,000) rounds
  t T_c / T half to even, in exact integer arithmetic.

Parity pins for every function live in ``tests/test_oracle_pins.py``.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Optional

import numpy as np
import scipy.linalg

__all__ = [
    "OracleConfig", "indexer_param_count", "rms_normalize", "value_context",
    "indexer_projections", "indexer_logits", "indexer_pool", "top_t", "CHUNK_THRESHOLD", "joint_compact_attention",
    "round_half_even_ratio", "chunk_budgets", "anchor_count", "top_t_chunked", "SELECTOR_EPS", "ha_scores",
    "leave_one_out_changes", "vi_scores", "truncated_output_error",
    "attention_logits", "full_attention", "response_profiles", "response_profiles_literal",
    "assign_to_anchors", "log_mass_weights", "mass_weights_literal", "merge_keys", "fit_beta", "fit_values", "compact_attention",
    "hard_subset_attention", "output_loss", "mass_error", "compact_pair", "compact_pair_steps",
]


@dataclasses.dataclass
class OracleConfig:
    t: int
    lambda_m: float = 0.25        # Sec. 4.1: 0.25 on QuALITY / RULER
    scale: Optional[float] = None  # None -> 1/sqrt(d)
    ridge_w: float = 1e-4
    ridge_v: float = 1e-3
    eps_w: float = float(np.exp(-20.0))
    b_min: float = -20.0
    b_max: float = 20.0
    G: int = 4
    chunk_len: int = 0             # App. A.3 fixed chunking (0: global top-t)
    selector: str = "indexer"      # "indexer" (Sec. 3.3), or "ha" / "vi" (App. B.1)


# ---------------------------------------------------------------- indexer

def indexer_param_count(d: int, d_x: int, H_I: int = 8, d_I: int = 128, d_A: int = 128) -> int:
    """Trainable parameters of one pair's indexer: Eqs. (indexer_parameters),
    (value_indexer_parameters) -- L_q, L_k in R^{H_I d_I x d}, L_x in
    R^{H_I x d_x}, b_x in R^{H_I}; U_q, U_k, U_v in R^{d_A x d},
    L_c in R^{H_I d_I x d_A}, L_v in R^{H_I d_I x d}."""
    HD = H_I * d_I
    return 2 * HD * d + H_I * d_x + H_I + 3 * d_A * d + HD * d_A + HD * d


def rms_normalize(z: np.ndarray, d_I: int) -> np.ndarray:
    """N(z) = z / sqrt(||z||^2 / d_I + 1e-6), applied to the last axis (App. A.1)."""
    return z / np.sqrt(np.sum(z * z, axis=-1, keepdims=True) / d_I + 1e-6)


def _softmax_rows(a: np.ndarray) -> np.ndarray:
    e = np.exp(a - a.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def value_context(Q, K, V, U_q, U_k, U_v):
    """Eq. (value_context): A^V_ij = softmax_j((U_q q_i).(U_k k_j)), c_i = sum_j A^V_ij U_v v_j.
    Returns (A^V [n,T], c [n,d_A])."""
    logits = (Q @ U_q.T) @ (K @ U_k.T).T
    A = _softmax_rows(logits)
    c = A @ (V @ U_v.T)
    return A, c


def indexer_projections(Q, X_rows, K, V, W, H_I: int = 8, d_I: int = 128):
    """Eq. (indexer_projection): q_bar [n,H_I,d_I], k_bar [T,H_I,d_I], w [n,H_I].

    ``X_rows`` is [n, d_x]: row i holds x_r of the reference position of row i.
    ``W`` maps names of App. A.1 to float64 arrays.
    """
    _, c = value_context(Q, K, V, W["U_q"], W["U_k"], W["U_v"])
    qz = (Q @ W["L_q"].T + c @ W["L_c"].T).reshape(Q.shape[0], H_I, d_I)
    kz = (K @ W["L_k"].T + V @ W["L_v"].T).reshape(K.shape[0], H_I, d_I)
    q_bar = rms_normalize(qz, d_I)
    k_bar = rms_normalize(kz, d_I)
    w = X_rows @ W["L_x"].T + W["b_x"][None, :]
    return q_bar, k_bar, w, c


def _run_steps(steps):
    """Run a step generator (below) to its end and return its result."""
    while True:
        try:
            next(steps)
        except StopIteration as done:
            return done.value


def _indexer_logits_steps(Q, X_rows, K, V, W, H_I: int = 8, d_I: int = 128):
    """indexer_logits one index head at a time: yields after the projections
    and after each head's term, returns I."""
    q_bar, k_bar, w, _ = indexer_projections(Q, X_rows, K, V, W, H_I, d_I)
    I = np.zeros((Q.shape[0], K.shape[0]))
    yield
    for a in range(H_I):
        x = (q_bar[:, a, :] @ k_bar[:, a, :].T) / np.sqrt(d_I)
        I += w[:, a:a + 1] * np.where(x >= 0.0, x, 0.1 * x)
        yield
    return I


def indexer_logits(Q, X_rows, K, V, W, H_I: int = 8, d_I: int = 128) -> np.ndarray:
    """Eq. (pairwise_index_score):
    I_ij = sum_a w_ia LeakyReLU_0.1(q_bar_ia . k_bar_ja / sqrt(d_I))."""
    return _run_steps(_indexer_logits_steps(Q, X_rows, K, V, W, H_I, d_I))


def indexer_pool(I: np.ndarray):
    """Eq. (indexer_pooling): pi = row softmax of I; s_j = (mean_i pi_ij^2)^(1/2).
    Returns (pi [n,T], s [T])."""
    pi = _softmax_rows(I)
    s = np.sqrt(np.mean(pi * pi, axis=0))
    return pi, s


def top_t(s: np.ndarray, t: int) -> np.ndarray:
    """Eq. (persistent_support): the t positions of largest s (ties -> lower
    position), returned in ascending position order."""
    order = np.lexsort((np.arange(s.shape[0]), -s))
    return np.sort(order[:t]).astype(np.int64)


CHUNK_THRESHOLD = 10_000   # App. A.3: fixed chunking applies only when T_a > 10,000


def round_half_even_ratio(num: int, den: int) -> int:
    """round(num / den) for integers num >= 0, den > 0, a tie going to the even
    neighbour; exact integer arithmetic (App. A.3 rounds t T_c / T_a)."""
    q, r = divmod(int(num), int(den))
    if 2 * r > den or (2 * r == den and q % 2 == 1):
        q += 1
    return q


def chunk_budgets(T: int, t: int, chunk_len: int, threshold: int = CHUNK_THRESHOLD):
    """App. A.3: with fixed chunking enabled (chunk_len > 0) and T_a = T above
    the threshold, the score vector is cut into contiguous chunks of length
    chunk_len (the last one shorter) and chunk c keeps
    t_c = clip_[1, T_c](round(t T_c / T)) anchors.  Returns [(start, T_c, t_c)];
    a single global chunk when chunking is off or bypassed."""
    if chunk_len <= 0 or T <= threshold:
        return [(0, T, t)]
    out = []
    for start in range(0, T, chunk_len):
        Tc = min(chunk_len, T - start)
        out.append((start, Tc, min(max(round_half_even_ratio(t * Tc, T), 1), Tc)))
    return out


def anchor_count(T: int, t: int, chunk_len: int, threshold: int = CHUNK_THRESHOLD) -> int:
    """Realized |S| = sum_c t_c (App. A.3: may differ slightly from t)."""
    return sum(tc for _, _, tc in chunk_budgets(T, t, chunk_len, threshold))


def top_t_chunked(s: np.ndarray, t: int, chunk_len: int, threshold: int = CHUNK_THRESHOLD) -> np.ndarray:
    """App. A.3: the union over chunks of each chunk's local top-t_c (ties ->
    lower position), in ascending position order."""
    parts = [start + top_t(s[start:start + Tc], tc) for start, Tc, tc in chunk_budgets(s.shape[0], t, chunk_len, threshold)]
    return np.concatenate(parts).astype(np.int64)


# ------------------------------------------------------- attention / merge

def attention_logits(Q, K, scale: float) -> np.ndarray:
    """Model-attention logits l_ij = scale * q_i . k_j (Sec. 3.1 with the scale reading)."""
    return scale * (Q @ K.T)


def full_attention(Q, K, V, scale: float):
    """Eq. (full_attention): P = softmax(QK^T), O = P V.  Returns (P, O)."""
    P = _softmax_rows(attention_logits(Q, K, scale))
    return P, P @ V


def response_profiles(l: np.ndarray):
    """Eq. (response_profile): u_j = exp(l_:j - z_merge) / ||exp(l_:j - z_merge)||_2
    with z_merge = max_ij l_ij.  Column j carries the common factor
    exp(M_j - z_merge), M_j = max_i l_ij, which the normalisation cancels, so
    the column is evaluated as exp(l_:j - M_j) / ||.|| -- the same vector,
    without the underflow of exp(l - z_merge) that fp64 meets once the logit
    range exceeds ~745.  Returns (u [n,T] with unit columns, M [T])."""
    M = l.max(axis=0)
    E = np.exp(l - M[None, :])
    return E / np.linalg.norm(E, axis=0, keepdims=True), M


def response_profiles_literal(l: np.ndarray):
    """Eq. (response_profile) with the single global shift z_merge, as printed
    (valid while the logit range stays inside fp64's exponent range)."""
    E = np.exp(l - l.max())
    return E / np.linalg.norm(E, axis=0, keepdims=True)


def _assign_steps(u: np.ndarray, S: np.ndarray, rows: int = 8192):
    """assign_to_anchors a block of keys at a time: yields after each block,
    returns kappa."""
    T = u.shape[1]
    uS = u[:, S]
    kappa = np.empty(T, dtype=np.int64)
    for j0 in range(0, T, rows):
        sim = u[:, j0:j0 + rows].T @ uS           # [rows, t]
        kappa[j0:j0 + rows] = np.argmax(sim, axis=1)  # first maximum = smallest r
        yield
    kappa[S] = np.arange(S.shape[0])
    return kappa


def assign_to_anchors(u: np.ndarray, S: np.ndarray, rows: int = 8192) -> np.ndarray:
    """Eq. (anchor_assignment): kappa(s_r) = r; kappa(j) = argmax_r u_j . u_{s_r}
    for j not in S (ties -> smallest r).  Each key's argmax is independent, so
    the T x t similarity table is formed ``rows`` keys at a time."""
    return _run_steps(_assign_steps(u, S, rows))


def log_mass_weights(l: np.ndarray) -> np.ndarray:
    """Eq. (mass_centroid): phi_j = (1/n) sum_i exp(l_ij - z_merge), returned as
    log phi_j + z_merge = M_j + log((1/n) sum_i exp(l_ij - M_j)).  The constant
    z_merge cancels in every ratio phi_j / sum_{G_r} phi that the merge uses."""
    M = l.max(axis=0)
    return M + np.log(np.mean(np.exp(l - M[None, :]), axis=0))


def mass_weights_literal(l: np.ndarray) -> np.ndarray:
    """Eq. (mass_centroid) as printed, phi_j = (1/n) sum_i exp(l_ij - z_merge)."""
    return np.exp(l - l.max()).mean(axis=0)


def merge_keys(K, kappa, logphi, S, lambda_m: float):
    """Eqs. (mass_centroid), (key_merge): mu_r = sum_{G_r} phi_j k_j / sum_{G_r} phi_j;
    c_{k,r} = (1 - lambda_m) k_{s_r} + lambda_m mu_r.  ``logphi`` is log phi up
    to a constant; each group's weights are scaled by exp(-max_{G_r} log phi),
    which cancels in the ratio.  Returns (C_k, mu)."""
    t = S.shape[0]
    gmax = np.full(t, -np.inf)
    np.maximum.at(gmax, kappa, logphi)
    wts = np.exp(logphi - gmax[kappa])
    num = np.zeros((t, K.shape[1]))
    den = np.zeros(t)
    np.add.at(num, kappa, wts[:, None] * K)
    np.add.at(den, kappa, wts)
    mu = num / den[:, None]
    return (1.0 - lambda_m) * K[S] + lambda_m * mu, mu


# ------------------------------------------------------------------- fits

def _ridge_solve(Gram: np.ndarray, rhs: np.ndarray, ridge: float) -> np.ndarray:
    """(Gram + lam I) x = rhs with lam = ridge * tr(Gram) / t, by Cholesky."""
    t = Gram.shape[0]
    lam = ridge * np.trace(Gram) / t
    A = Gram + lam * np.eye(t)
    c, low = scipy.linalg.cho_factor(A, lower=True, check_finite=True)
    return scipy.linalg.cho_solve((c, low), rhs)


def fit_beta(Q, K, C_k, cfg: OracleConfig, scale: float):
    """Eq. (mass_fit): z_i = max_j q_i.k_j; Phi_K = exp(QK^T - z), Phi_C =
    exp(QC_k^T - z); w~ = argmin ||Phi_C w - Phi_K 1||^2 (ridge reading);
    w* = max(w~, 0); beta = clip(log max(w*, eps_w), b_min, b_max).
    Returns dict(beta, w_tilde, w_star, Phi_C, Phi_K_row_mass, z)."""
    l = attention_logits(Q, K, scale)
    z = l.max(axis=1)
    Phi_K = np.exp(l - z[:, None])
    Phi_C = np.exp(attention_logits(Q, C_k, scale) - z[:, None])
    m = Phi_K.sum(axis=1)
    w_tilde = _ridge_solve(Phi_C.T @ Phi_C, Phi_C.T @ m, cfg.ridge_w)
    w_star = np.maximum(w_tilde, 0.0)
    beta = np.clip(np.log(np.maximum(w_star, cfg.eps_w)), cfg.b_min, cfg.b_max)
    return {"beta": beta, "w_tilde": w_tilde, "w_star": w_star, "Phi_C": Phi_C, "m": m, "z": z}


def fit_values(Q, K, V, C_k, beta, cfg: OracleConfig, scale: float):
    """Eq. (value_lstsq): P^ = softmax(Q C_k^T + 1 beta^T), Y = softmax(QK^T) V,
    C_v = argmin ||P^ C - Y||_F^2 + lam_v ||C||_F^2.  Returns dict(C_v, P_hat, Y)."""
    P_hat = _softmax_rows(attention_logits(Q, C_k, scale) + beta[None, :])
    _, Y = full_attention(Q, K, V, scale)
    C_v = _ridge_solve(P_hat.T @ P_hat, P_hat.T @ Y, cfg.ridge_v)
    return {"C_v": C_v, "P_hat": P_hat, "Y": Y}


def compact_attention(Q, C_k, beta, C_v, scale: float) -> np.ndarray:
    """Eq. (compact_attention): O^ = softmax(Q C_k^T + 1 beta^T) C_v."""
    return _softmax_rows(attention_logits(Q, C_k, scale) + beta[None, :]) @ C_v


def joint_compact_attention(Q, C_k, beta, C_v, K_fixed, V_fixed, scale: float) -> np.ndarray:
    """Eq. (concatenated_attention_preservation), right-hand side: attention
    over the stacked keys [C_k; K_fixed] and values [C_v; V_fixed] with the
    bias b = [beta; 0_F] on the logits (App. A.7).  Either block may be empty."""
    keys = np.concatenate([C_k, K_fixed], axis=0)
    vals = np.concatenate([C_v, V_fixed], axis=0)
    b = np.concatenate([beta, np.zeros(K_fixed.shape[0])])
    return _softmax_rows(attention_logits(Q, keys, scale) + b[None, :]) @ vals


def hard_subset_attention(Q, K, V, S, scale: float) -> np.ndarray:
    """Eq. (background_hard_attention): softmax(q K_S^T) V_S."""
    return _softmax_rows(attention_logits(Q, K[S], scale)) @ V[S]


# ------------------------------------------------- HA / VI selectors, E(S)

SELECTOR_EPS = 1e-6   # the epsilon of Eqs. background_value_selectors / background_truncated_error (unstated)


def ha_scores(Q, K, scale: float) -> np.ndarray:
    """App. B.1 Eq. (background_value_selectors): s^HA_j = (mean_i p_ij^2)^(1/2),
    p = softmax(scale Q K^T)."""
    P = _softmax_rows(attention_logits(Q, K, scale))
    return np.sqrt(np.mean(P * P, axis=0))


def leave_one_out_changes(Q, K, V, scale: float) -> np.ndarray:
    """D_ij = ||O_i - O_i^(-j)|| = p_ij / (1 - p_ij) ||v_j - O_i|| (App. B.1), with
    1 - p_ij = sum_{u != j} p_iu.  For the column a_i holding a row's largest
    logit the same quantity is evaluated as p_ia ||v_a - O_i^(-a)|| (exact
    algebra: O_i = p_ia v_a + (1 - p_ia) O_i^(-a)), O_i^(-a) being attention over
    the other keys with its own max shift -- where p_ia rounds to 1 and v_a to
    O_i, the printed form is 0 / 0 in any floating point."""
    l = attention_logits(Q, K, scale)
    n, T = l.shape
    z = l.max(axis=1, keepdims=True)
    e = np.exp(l - z)
    msum = e.sum(axis=1, keepdims=True)
    O = (e @ V) / msum
    # non-dominant columns: p / (1 - p) = e / (sum_{u != j} e_u)
    vv = np.sum(V * V, axis=1)[None, :]
    oo = np.sum(O * O, axis=1)[:, None]
    dist2 = np.maximum(vv - 2.0 * (O @ V.T) + oo, 0.0)
    a = np.argmax(l, axis=1)
    den = msum - e
    den[np.arange(n), a] = 1.0          # the dominant columns are evaluated below
    D = e / den * np.sqrt(dist2)
    for i in range(n):
        rest = np.delete(np.arange(T), a[i])
        if rest.size == 0:
            D[i, a[i]] = np.inf
            continue
        lr = l[i, rest]
        z2 = lr.max()
        er = np.exp(lr - z2)
        O_minus = (er @ V[rest]) / er.sum()
        p_a = 1.0 / (1.0 + er.sum() * np.exp(z2 - z[i, 0]))
        D[i, a[i]] = p_a * np.linalg.norm(V[a[i]] - O_minus)
    return D


def vi_scores(Q, K, V, scale: float, eps: float = SELECTOR_EPS) -> np.ndarray:
    """App. B.1 Eq. (background_value_selectors):
    s^VI_j = (mean_i D_ij^2 / (||O_i||^2 + eps))^(1/2)."""
    D = leave_one_out_changes(Q, K, V, scale)
    O = full_attention(Q, K, V, scale)[1]
    oo = np.sum(O * O, axis=1)[:, None]
    return np.sqrt(np.mean(D * D / (oo + eps), axis=0))


def truncated_output_error(Q_eval, K, V, S, scale: float, eps: float = SELECTOR_EPS) -> float:
    """App. B.1 Eq. (background_truncated_error): O~_i(S) = sum_{j in S} p_ij v_j
    with p, O from the full cache; E(S) = mean_i ||O_i - O~_i|| / (||O_i|| + eps)."""
    P, O = full_attention(Q_eval, K, V, scale)
    S = np.asarray(S, dtype=np.int64)
    O_t = P[:, S] @ V[S]
    return float(np.mean(np.linalg.norm(O - O_t, axis=1) / (np.linalg.norm(O, axis=1) + eps)))


# ------------------------------------------------------------ diagnostics

def output_loss(y_hat: np.ndarray, y: np.ndarray) -> float:
    """Eq. (output_loss): mean_i ||y^_i - y_i||^2 / ||y_i||^2."""
    return float(np.mean(np.sum((y_hat - y) ** 2, axis=1) / np.sum(y * y, axis=1)))


def mass_error(Phi_C: np.ndarray, w_star: np.ndarray, m: np.ndarray) -> float:
    """App. E.1: E_mass = ||Z_c - Z_f|| / ||Z_f||, Z_f = Phi_K 1, Z_c = Phi_C w*."""
    return float(np.linalg.norm(Phi_C @ w_star - m) / np.linalg.norm(m))


# --------------------------------------------------------------- pipeline

def compact_pair_steps(K, V, Q, X_rows, W, cfg: OracleConfig, anchors_in: Optional[np.ndarray] = None,
                       assign_in: Optional[np.ndarray] = None, H_I: int = 8, d_I: int = 128):
    """compact_pair as a sequence of bounded steps: a generator that yields
    between stages (and between index heads and key blocks inside the two
    longest) and returns compact_pair's result.  The arithmetic is
    compact_pair's; only the points where it may pause are added, so that a
    caller can time the pipeline piece by piece."""
    d = K.shape[1]
    scale = cfg.scale if cfg.scale is not None else 1.0 / np.sqrt(d)
    out: Dict[str, np.ndarray] = {}
    if anchors_in is None:
        if cfg.selector == "indexer":
            I = yield from _indexer_logits_steps(Q, X_rows, K, V, W, H_I, d_I)
            _, s = indexer_pool(I)
            del I
        elif cfg.selector == "ha":
            s = ha_scores(Q, K, scale)
        else:
            s = vi_scores(Q, K, V, scale)
        S = top_t_chunked(s, cfg.t, cfg.chunk_len)
        out["scores"] = s
        yield
    else:
        S = np.asarray(anchors_in, dtype=np.int64)
    l = attention_logits(Q, K, scale)
    u, _ = response_profiles(l)
    yield
    if assign_in is None:
        kappa = yield from _assign_steps(u, S)
    else:
        kappa = np.asarray(assign_in, dtype=np.int64)
    del u
    logphi = log_mass_weights(l)
    del l
    C_k, _ = merge_keys(K, kappa, logphi, S, cfg.lambda_m)
    yield
    fb = fit_beta(Q, K, C_k, cfg, scale)
    yield
    fv = fit_values(Q, K, V, C_k, fb["beta"], cfg, scale)
    out.update(anchors=S, assign=kappa, logphi=logphi, C_k=C_k, beta=fb["beta"],
               w_star=fb["w_star"], w_tilde=fb["w_tilde"], C_v=fv["C_v"],
               mass_error=mass_error(fb["Phi_C"], fb["w_star"], fb["m"]))
    return out


def compact_pair(K, V, Q, X_rows, W, cfg: OracleConfig, anchors_in: Optional[np.ndarray] = None,
                 assign_in: Optional[np.ndarray] = None, H_I: int = 8, d_I: int = 128) -> Dict[str, np.ndarray]:
    """One layer-KV-head pair through the four stages of Sec. 3.2:
    indexer scoring and top-t (Sec. 3.3), response-profile assignment and
    convex key merge (Sec. 3.4), then the beta and C_v fits (App. A.9).
    ``anchors_in`` replaces the scored anchor set (the hard-branch setting of
    Sec. 3.5, also used to compare stages downstream of selection);
    ``assign_in`` likewise replaces the computed assignment."""
    return _run_steps(compact_pair_steps(K, V, Q, X_rows, W, cfg, anchors_in, assign_in, H_I, d_I))
