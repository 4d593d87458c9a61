"""Comparison helpers for GPU-vs-oracle parity (test infrastructure only).

Tolerances (applied by the tests, stated here once):
  * pooled scores: ||s_gpu - s||_inf / ||s||_inf <= 1e-3, and elementwise
    relative error <= 1e-3 on the oracle's top-2t scores;
  * anchor sets: identical, except that positions whose oracle score lies
    within ``band`` (relative to the oracle's t-th largest score) of that
    threshold may be exchanged for one another (a tie band).  The band may be
    widened by the GPU scores' own relative errors at the position and at the
    t-th key -- top-t cannot order keys closer than the errors of the scores
    that rank them -- but only while those two errors add up to no more than
    ``WIDEN_CAP`` (2e-5), so an exchange is never accepted beyond
    band + 2e-5; with chunked selection the same holds within each chunk at
    its own t_c-th score;
  * assignment (an argmax whose exact ties are frequent): where the oracle's
    best and second-best similarities differ by more than ``tau`` the GPU
    must agree; elsewhere the GPU's choice must be within ``tau`` of the best;
  * C_k, C_v, held-out outputs: relative Frobenius error <= 2e-3;
  * beta: relative l2 error <= 2e-3 over entries whose oracle w* exceeds
    1e-6 max w*; on the remaining entries the GPU's beta must also sit at a
    near-zero weight (beta <= log(1e-5 max w*)).  For anchor sets whose mass
    fit is too ill-conditioned for that in fp32 (the HA / VI selectors of
    App. B.1: Phi_C columns spanning four decades), beta is compared as the
    mass weights e^beta it contributes to Eq. compact_attention: relative l2
    <= 2e-3 (mass_weight_error).
"""
from __future__ import annotations

import numpy as np


def rel_inf(a, b) -> float:
    return float(np.max(np.abs(a - b)) / np.max(np.abs(b)))


def rel_fro(a, b) -> float:
    nb = float(np.linalg.norm(b))
    return float(np.linalg.norm(a - b) / (nb if nb > 0 else 1.0))


def score_errors(s_gpu: np.ndarray, s: np.ndarray, t: int):
    """(inf-norm relative error, max elementwise relative error on the top-2t)."""
    top = np.argsort(-s, kind="stable")[: min(len(s), 2 * t)]
    return rel_inf(s_gpu, s), float(np.max(np.abs(s_gpu[top] - s[top]) / np.abs(s[top])))


WIDEN_CAP = 2e-5   # largest sum of GPU score errors that may widen the anchor tie band


def anchors_match(S_gpu: np.ndarray, S: np.ndarray, s: np.ndarray, t: int, band: float, s_gpu=None):
    """True if the anchor sets agree up to exchanges inside the tie band.

    Top-t keeps the t largest scores; a key can only enter or leave the set
    through an error of the scores that decided it.  An exchanged position j
    is accepted when its oracle score lies within ``band`` (relative) of the
    oracle's t-th score.  When the GPU scores ``s_gpu`` are given, the band
    at j is widened by the GPU's relative errors at j and at the t-th key
    (the two keys' order is not fixed by scores carrying those errors),
    provided those errors add up to at most WIDEN_CAP; larger errors widen
    nothing.  Returns (ok, number of exchanged positions, widest relative gap
    |s_j - s_(t)| / s_(t) among the exchanged positions)."""
    order = np.argsort(-s, kind="stable")
    k_thr = int(order[t - 1])
    thr = s[k_thr]
    a, b = set(map(int, S_gpu)), set(map(int, S))
    diff = sorted(a ^ b)
    if len(a) != len(b) or len(S_gpu) != t:
        return False, len(diff), float("inf")
    if not diff:
        return True, 0, 0.0

    def err(j):
        return 0.0 if s_gpu is None else abs(float(s_gpu[j]) - s[j]) / abs(s[j])

    def widen(j):
        w = err(j) + err(k_thr)
        return w if w <= WIDEN_CAP else 0.0

    gaps = [abs(s[j] - thr) / thr for j in diff]
    ok = all(g <= band + widen(j) for g, j in zip(gaps, diff))
    return bool(ok), len(diff), float(max(gaps))


def anchors_match_chunked(S_gpu: np.ndarray, S: np.ndarray, s: np.ndarray, chunks, band: float, s_gpu=None):
    """anchors_match within every chunk (start, T_c, t_c) of the chunked
    selection of App. A.3, the tie band taken at the chunk's own t_c-th score.
    Returns (ok, exchanged positions, widest relative gap)."""
    n_ex, widest = 0, 0.0
    for start, Tc, tc in chunks:
        def part(X):
            X = np.asarray(X)
            return X[(X >= start) & (X < start + Tc)] - start
        sg = None if s_gpu is None else s_gpu[start:start + Tc]
        ok, nd, gap = anchors_match(part(S_gpu), part(S), s[start:start + Tc], tc, band, sg)
        if not ok:
            return False, nd, gap
        n_ex += nd
        widest = max(widest, gap)
    return len(S_gpu) == len(S), n_ex, widest


def assignment_valid(kappa_gpu: np.ndarray, sim: np.ndarray, S: np.ndarray, tau: float):
    """Check a GPU assignment against the oracle's similarity table sim [T, t].
    Returns (ok, n_decided_mismatch, n_tied_differences, worst shortfall)."""
    T = sim.shape[0]
    best = sim.max(axis=1)
    srt = np.sort(sim, axis=1)
    gap = srt[:, -1] - (srt[:, -2] if sim.shape[1] > 1 else -np.inf)
    is_anchor = np.zeros(T, bool)
    is_anchor[S] = True
    got = sim[np.arange(T), kappa_gpu]
    short = best - got
    dec = (~is_anchor) & (gap > tau)
    kappa_ref = np.argmax(sim, axis=1)
    n_dec_mis = int(np.sum(dec & (kappa_gpu != kappa_ref)))
    anchors_ok = bool(np.all(kappa_gpu[S] == np.arange(len(S))))
    worst = float(np.max(np.where(is_anchor, 0.0, short)))
    n_tie = int(np.sum((~is_anchor) & (~dec) & (kappa_gpu != kappa_ref)))
    return (n_dec_mis == 0 and anchors_ok and worst <= tau), n_dec_mis, n_tie, worst


def assignment_valid_profiles(kappa_gpu: np.ndarray, u: np.ndarray, S: np.ndarray, tau: float, rows: int = 8192):
    """assignment_valid over the profile matrix u [n, T], forming the
    similarity table a block of keys at a time (for long caches)."""
    T = u.shape[1]
    uS = u[:, S]
    is_anchor = np.zeros(T, bool)
    is_anchor[S] = True
    n_mis = n_tie = 0
    worst = 0.0
    for j0 in range(0, T, rows):
        sim = u[:, j0:j0 + rows].T @ uS
        kg = kappa_gpu[j0:j0 + rows]
        best = sim.max(axis=1)
        srt = np.sort(sim, axis=1)
        gap = srt[:, -1] - (srt[:, -2] if sim.shape[1] > 1 else -np.inf)
        anc = is_anchor[j0:j0 + rows]
        got = sim[np.arange(sim.shape[0]), kg]
        dec = (~anc) & (gap > tau)
        kref = np.argmax(sim, axis=1)
        n_mis += int(np.sum(dec & (kg != kref)))
        n_tie += int(np.sum((~anc) & (~dec) & (kg != kref)))
        worst = max(worst, float(np.max(np.where(anc, 0.0, best - got))))
    anchors_ok = bool(np.all(kappa_gpu[S] == np.arange(len(S))))
    return (n_mis == 0 and anchors_ok and worst <= tau), n_mis, n_tie, worst


def beta_errors(beta_gpu: np.ndarray, beta: np.ndarray, w_star: np.ndarray):
    """(relative l2 error on the supported entries, ok flag for the rest)."""
    wmax = float(np.max(w_star))
    sup = w_star > 1e-6 * wmax
    e = rel_fro(beta_gpu[sup], beta[sup]) if np.any(sup) else 0.0
    rest_ok = bool(np.all(beta_gpu[~sup] <= np.log(max(1e-5 * wmax, 1e-300)) + 1e-6))
    return e, rest_ok


def mass_weight_error(beta_gpu: np.ndarray, beta: np.ndarray) -> float:
    """Relative l2 error of the mass weights e^beta (the factor beta puts on
    each compact key's attention weight in Eq. compact_attention)."""
    return rel_fro(np.exp(np.asarray(beta_gpu, dtype=np.float64)), np.exp(np.asarray(beta, dtype=np.float64)))
