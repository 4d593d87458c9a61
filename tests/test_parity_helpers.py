"""The GPU-vs-oracle comparison helpers (``oracle/parity.py``) on constructed
cases whose outcome is known: a checker that accepts everything would make
every GPU parity test vacuous, one that rejects valid results would hide
real agreement.  CPU only."""
import numpy as np

from oracle import parity


def test_relative_norms():
    b = np.array([3.0, -4.0])
    assert np.isclose(parity.rel_fro(b + np.array([0.3, 0.4]), b), 0.1, rtol=1e-14)
    assert np.isclose(parity.rel_inf(b + np.array([0.0, 0.4]), b), 0.1, rtol=1e-14)
    assert np.isclose(parity.rel_fro(np.ones(3), np.zeros(3)), np.sqrt(3.0), rtol=1e-14)   # zero reference: absolute norm


def test_score_errors_inf_norm_and_top_2t():
    s = np.array([10.0, 1.0, 8.0, 2.0, 0.5, 9.0])
    g = s.copy()
    g[1] *= 1.2          # not among the top 2t = 4 (10, 9, 8, 2): only the inf-norm sees it
    e_inf, e_top = parity.score_errors(g, s, 2)
    assert np.isclose(e_inf, 0.02, rtol=1e-12) and e_top == 0.0
    g[3] *= 1.01         # 4th largest: inside the top 2t
    assert np.isclose(parity.score_errors(g, s, 2)[1], 0.01, rtol=1e-12)


def test_anchors_identical_and_wrong_size():
    s = np.linspace(1.0, 2.0, 10)
    S = np.arange(5, 10)
    assert parity.anchors_match(S, S, s, 5, 1e-5) == (True, 0, 0.0)
    ok, _, gap = parity.anchors_match(S[:4], S, s, 5, 1e-5)
    assert not ok and gap == float("inf")


def test_anchor_exchange_inside_and_outside_the_band():
    s = np.array([5.0, 4.0, 3.0, 2.0 + 1e-6, 2.0, 1.0])   # t = 4: threshold 2 + 1e-6 (position 3)
    S = np.array([0, 1, 2, 3])
    near = np.array([0, 1, 2, 4])                         # key 4 sits 5e-7 (relative) below the threshold
    ok, nd, gap = parity.anchors_match(near, S, s, 4, 1e-5)
    assert ok and nd == 2 and gap < 1e-6
    far = np.array([0, 1, 3, 5])                          # key 5 is half the threshold away
    ok, nd, gap = parity.anchors_match(far, S, s, 4, 1e-5)
    assert not ok and gap > 0.4
    # the band is measured from the t-th score itself: keys 8e-6 above and below
    # it may trade places (band 1e-5), though they lie 1.6e-5 apart
    s = np.array([5.0, 2.0 * (1 + 8e-6), 2.0, 2.0 * (1 - 8e-6), 1.0])
    assert parity.anchors_match(np.array([0, 2, 3]), np.array([0, 1, 2]), s, 3, 1e-5)[0]


def test_anchor_band_widened_by_the_gpu_score_errors():
    thr = 2.0
    s = np.array([5.0, 4.0, 3.0, thr, thr * (1 - 2.5e-5), 1.0])
    S = np.array([0, 1, 2, 3])
    swapped = np.array([0, 1, 2, 4])
    assert not parity.anchors_match(swapped, S, s, 4, 1e-5)[0]          # 2.5e-5 > band
    g = s.copy()
    g[4] *= 1 + 1.8e-5   # the GPU's score at key 4 carries a 1.8e-5 error: 2.5e-5 - 1.8e-5 <= 1e-5
    ok, nd, gap = parity.anchors_match(swapped, S, s, 4, 1e-5, g)
    assert ok and nd == 2 and np.isclose(gap, 2.5e-5, rtol=1e-9)      # the widest accepted gap is reported
    g = s.copy()
    g[4] *= 1 + 1e-5     # too small an error to explain a 2.5e-5 gap
    assert not parity.anchors_match(swapped, S, s, 4, 1e-5, g)[0]
    g = s.copy()
    g[3] *= 1 - 1.8e-5   # the error may sit at the t-th key instead
    assert parity.anchors_match(swapped, S, s, 4, 1e-5, g)[0]
    # errors above the cap (2e-5 in total) widen nothing: a GPU whose scores are
    # that far off cannot excuse an exchange beyond the plain band
    g = s.copy()
    g[4] *= 1 + 3e-5
    assert not parity.anchors_match(swapped, S, s, 4, 1e-5, g)[0]
    g = s.copy()
    g[4] *= 1 + 1.2e-5
    g[3] *= 1 - 1.2e-5   # 2.4e-5 in total: above the cap
    assert not parity.anchors_match(swapped, S, s, 4, 1e-5, g)[0]
    assert parity.WIDEN_CAP == 2e-5


def test_chunked_anchors_keep_each_chunk_to_its_own_budget():
    s = np.array([4.0, 3.0, 2.0, 1.0, 4.0, 3.0, 2.0, 1.0 + 1e-7])
    chunks = [(0, 4, 2), (4, 4, 2)]
    S = np.array([0, 1, 4, 5])
    assert parity.anchors_match_chunked(S, S, s, chunks, 1e-5)[0]
    # a key moved from chunk 0 to chunk 1: the union has the right size but
    # neither chunk keeps its own budget
    moved = np.array([0, 4, 5, 6])
    assert not parity.anchors_match_chunked(moved, S, s, chunks, 1e-5)[0]
    # inside chunk 1 an exchange at a near tie is accepted only within its band
    s2 = s.copy(); s2[6] = 3.0 * (1 - 1e-6)
    ok, nd, _ = parity.anchors_match_chunked(np.array([0, 1, 4, 6]), S, s2, chunks, 1e-5)
    assert ok and nd == 2


def test_assignment_decided_and_tied_rows():
    # rows: keys, columns: anchors (anchors are keys 0 and 1)
    sim = np.array([[1.0, 0.2],
                    [0.2, 1.0],
                    [0.9, 0.3],            # decided: anchor 0
                    [0.50, 0.50 - 1e-6]])  # tied within tau = 1e-4
    S = np.array([0, 1])
    ok, n_mis, n_tie, worst = parity.assignment_valid(np.array([0, 1, 0, 1]), sim, S, 1e-4)
    assert ok and n_mis == 0 and n_tie == 1 and np.isclose(worst, 1e-6, rtol=1e-9)
    ok, n_mis, _, _ = parity.assignment_valid(np.array([0, 1, 1, 0]), sim, S, 1e-4)
    assert not ok and n_mis == 1
    ok = parity.assignment_valid(np.array([1, 1, 0, 0]), sim, S, 1e-4)[0]   # anchor 0 not mapped to itself
    assert not ok
    # three anchors, a row whose best two are tied: either of them is valid,
    # the distant third is not, though the row counts as undecided
    sim3 = np.array([[1.0, 0.1, 0.1], [0.1, 1.0, 0.1], [0.1, 0.1, 1.0], [0.5, 0.5 - 1e-6, 0.1]])
    S3 = np.array([0, 1, 2])
    assert parity.assignment_valid(np.array([0, 1, 2, 1]), sim3, S3, 1e-4)[0]
    ok, n_mis, _, worst = parity.assignment_valid(np.array([0, 1, 2, 2]), sim3, S3, 1e-4)
    assert not ok and n_mis == 0 and np.isclose(worst, 0.4)


def test_assignment_on_profiles_matches_the_table_form():
    rng = np.random.default_rng(3)
    u = rng.random((6, 40)); u /= np.linalg.norm(u, axis=0, keepdims=True)
    S = np.array([2, 11, 30])
    sim = u.T @ u[:, S]
    kappa = np.argmax(sim, axis=1); kappa[S] = np.arange(3)
    assert parity.assignment_valid_profiles(kappa, u, S, 1e-4, rows=7) == parity.assignment_valid(kappa, sim, S, 1e-4)
    j = next(j for j in range(40) if j not in S and np.sort(sim[j])[-1] - np.sort(sim[j])[-2] > 1e-3)
    bad = kappa.copy(); bad[j] = (bad[j] + 1) % 3
    assert not parity.assignment_valid_profiles(bad, u, S, 1e-4, rows=7)[0]


def test_beta_support_rule_and_mass_weights():
    w_star = np.array([2.0, 1.0, 1e-9, 0.0])
    beta = np.log(np.maximum(w_star, np.exp(-20.0)))
    g = beta.copy(); g[0] += 1e-3
    e, rest_ok = parity.beta_errors(g, beta, w_star)
    assert np.isclose(e, 1e-3 / np.linalg.norm(beta[:2])) and rest_ok
    g = beta.copy(); g[3] = np.log(1e-3)        # an unsupported anchor given real weight
    assert not parity.beta_errors(g, beta, w_star)[1]
    assert np.isclose(parity.mass_weight_error(np.log([2.0, 1.0]) + np.log(1.01), np.log([2.0, 1.0])), 0.01)
