"""The seeded input generator (``synth/``) against the recipe it states:
properties of the drawn tensors, not a retyping of the generator.  CPU only."""
import numpy as np
import pytest
import torch

import synth

W = synth.WORKLOADS["llama8b_layer_T8192"]


def test_bf16_rounding_matches_torch_including_ties():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(4096) * 10.0 ** rng.integers(-6, 6, 4096)).astype(np.float32)
    # exact halfway cases: 1 + 2^-8 (between 1 and 1 + 2^-7; ties to the even 1.0)
    # and 1 + 3 * 2^-8 (ties to the even 1 + 2^-6)
    x = np.concatenate([x, np.float32([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 0.0, -0.0])])
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(synth.bf16_round(x), want)
    assert synth.bf16_to_f64(synth.bf16_round(np.float32([1 + 2 ** -8])))[0] == 1.0


def test_rope_is_a_rotation_with_relative_position_dot_products():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((6, 128))
    pos = np.array([0, 1, 7, 100, 4096, 8191])
    r = synth._rope(x, pos)
    half = 64
    # each channel pair (i, i + 64) is rotated: its energy is kept
    assert np.allclose(r[:, :half] ** 2 + r[:, half:] ** 2, x[:, :half] ** 2 + x[:, half:] ** 2, rtol=1e-12)
    assert np.array_equal(r[0], x[0])                          # position 0: identity
    # pair 0 turns by exactly the position (inverse frequency theta^0 = 1)
    ang = np.arctan2(r[:, half], r[:, 0]) - np.arctan2(x[:, half], x[:, 0])
    assert np.allclose(np.cos(ang), np.cos(pos), atol=1e-9) and np.allclose(np.sin(ang), np.sin(pos), atol=1e-9)
    # the last pair turns at theta^(-126/128) per position, theta = 500000
    e = np.zeros((1, 128)); e[0, 63] = 1.0
    re = synth._rope(e, np.array([1000]))
    assert np.isclose(np.arctan2(re[0, 127], re[0, 63]), 1000 * 500000.0 ** (-126 / 128), rtol=1e-12)
    # q(m) . k(n) depends on m - n only
    q, k = rng.standard_normal((1, 128)), rng.standard_normal((1, 128))
    a = synth._rope(q, np.array([10])) @ synth._rope(k, np.array([3])).T
    b = synth._rope(q, np.array([1007])) @ synth._rope(k, np.array([1000])).T
    assert np.isclose(a, b, rtol=1e-9)


def _pair_energy(K):
    k = synth.bf16_to_f64(K)
    return np.mean(k[1:, :64] ** 2 + k[1:, 64:] ** 2, axis=0)    # row 0 is the sink


def test_keys_outlier_channels_and_attention_sink():
    p = synth.make_pair(W, 0, 0, T=2048, n_pos=8)
    e = _pair_energy(p["K"])
    # four channels x 8 before RoPE: their pairs carry ~64 + 1 instead of 2
    hot = np.sort(e)[::-1]
    assert 2 <= np.sum(e > 20) <= 4
    assert 200 < np.sum(hot[:4]) - 2 * 4 < 330 and np.all(np.sort(e)[:-4] < 2.5)
    norms = np.linalg.norm(synth.bf16_to_f64(p["K"]), axis=1)
    assert 7.0 < norms[0] / np.median(norms[1:]) < 14.0      # x10 in norm (the row's own norm varies)


def test_outlier_channels_reseeded_per_layer_only_for_the_32k_workload():
    w32 = synth.WORKLOADS["llama8b_T32768_r05"]
    ch = lambda w, l: tuple(synth._outlier_channels(w, l))
    assert ch(W, 0) == ch(W, 5)
    assert len({ch(w32, l) for l in range(6)}) > 1


def test_values_queries_and_activations_follow_their_laws():
    p = synth.make_pair(W, 0, 1, T=1024, n_pos=64)
    v = synth.bf16_to_f64(p["V"])
    assert abs(v.mean()) < 0.02 and abs(v.var() - 1.0) < 0.03
    # values are drawn independently of the keys: matched channels are uncorrelated
    kk = synth.bf16_to_f64(p["K"])[1:]
    corr = [np.corrcoef(kk[:, c], v[1:, c])[0, 1] for c in range(128)]
    assert np.max(np.abs(corr)) < 0.15
    # each query is a key plus N(0, 0.5^2): its nearest key sits at squared distance ~0.25 per dim
    q, k = synth.bf16_to_f64(p["Q"]), synth.bf16_to_f64(p["K"])
    d2 = ((q[:, None, :] - k[None, :, :]) ** 2).sum(-1).min(1) / 128
    assert p["Q"].shape == (64 * W.G, 128) and 0.2 < np.median(d2) < 0.3
    x = synth.bf16_to_f64(synth.make_layer_activations(W, 0, n_pos=16))
    assert x.shape == (16, W.shape.d_x) and abs(x.std() - 1.0) < 0.02


def test_indexer_weight_scales_and_zero_value_path():
    idx = synth.make_indexer(W, 0, 0)
    s = W.shape
    std = lambda k: synth.bf16_to_f64(idx[k]).std()
    for k, want in (("U_q", s.d ** -0.5), ("L_k", s.d ** -0.5), ("L_c", s.d_A ** -0.5), ("L_x", s.d_x ** -0.5),
                    ("b_x", 0.1)):
        assert abs(std(k) / want - 1.0) < (0.5 if k == "b_x" else 0.05), k
    assert idx["L_q"].shape == (s.H_I * s.d_I, s.d) and idx["L_x"].shape == (s.H_I, s.d_x)
    z = synth.make_indexer(W, 0, 0, zero_value_path=True)
    assert not z["L_c"].any() and not z["L_v"].any() and np.array_equal(z["L_q"], idx["L_q"])


def test_pairs_regenerate_alone_and_differ_across_heads():
    a = synth.make_pair(W, 2, 3, T=256, n_pos=4)
    synth.make_pair(W, 0, 0, T=256, n_pos=4)
    b = synth.make_pair(W, 2, 3, T=256, n_pos=4)
    c = synth.make_pair(W, 2, 4, T=256, n_pos=4)
    assert all(np.array_equal(a[k], b[k]) for k in "KVQ")
    assert not np.array_equal(a["K"], c["K"]) and not np.array_equal(a["V"], c["V"])
    # a shorter T gives the first T rows of the same cache (one stream per tensor family)
    short = synth.make_pair(W, 2, 3, T=128, n_pos=4)
    assert np.array_equal(short["K"], a["K"][:128]) and np.array_equal(short["V"], a["V"][:128])


@pytest.mark.parametrize("name", sorted(synth.WORKLOADS))
def test_workload_table(name):
    w = synth.WORKLOADS[name]
    assert w.n == w.n_pos * w.G and 1 <= w.t <= w.T
    if "_r" in name:
        ratio = int(name.rsplit("_r", 1)[1]) / 100
        assert w.t == int(np.floor(ratio * w.T))      # t = floor(rho T)


def _device_layer(layer=0, heads=(0, 1), T=2048, n_pos=64):
    d = synth.make_layer_device(W, layer, list(heads), "cpu", T=T, n_pos=n_pos)
    bits = lambda t: t.contiguous().view(torch.int16).numpy().view(np.uint16)
    return {k: bits(v) for k, v in d.items()}


def test_device_layers_follow_the_same_recipe():
    """The device-side layer generator (used to time whole 128K contexts):
    the key, value and query laws of the host path, checked the same way."""
    d = _device_layer()
    assert d["K"].shape == (2, 2048, 128) and d["Q"].shape == (2, 64 * W.G, 128)
    e = _pair_energy(d["K"][0])
    assert 2 <= np.sum(e > 20) <= 4 and np.all(np.sort(e)[:-4] < 2.5)
    # the same outlier channels as the host path (their rotation pairs carry the energy)
    host_pairs = {c % 64 for c in synth._outlier_channels(W, 0)}
    assert set(np.argsort(e)[::-1][:len(host_pairs)]) == host_pairs
    norms = np.linalg.norm(synth.bf16_to_f64(d["K"][0]), axis=1)
    assert 7.0 < norms[0] / np.median(norms[1:]) < 14.0
    v = synth.bf16_to_f64(d["V"][0])
    assert abs(v.mean()) < 0.02 and abs(v.var() - 1.0) < 0.03
    kk = synth.bf16_to_f64(d["K"][0])[1:]
    assert max(abs(np.corrcoef(kk[:, c], v[1:, c])[0, 1]) for c in range(128)) < 0.15
    q, k = synth.bf16_to_f64(d["Q"][0]), synth.bf16_to_f64(d["K"][0])
    d2 = ((q[:, None, :] - k[None, :, :]) ** 2).sum(-1).min(1) / 128
    assert 0.2 < np.median(d2) < 0.3
    # the device rotation is the host's (float64 angles, float32 products)
    rng = np.random.default_rng(4)
    x = rng.standard_normal((5, 128)).astype(np.float32)
    pos = np.array([0, 3, 999, 65536, 131071])
    r_dev = synth._rope_torch(torch.from_numpy(x), torch.from_numpy(pos)).numpy()
    assert np.allclose(r_dev, synth._rope(x.astype(np.float64), pos), rtol=1e-5, atol=1e-5)
    host = synth.make_pair(W, 0, 0, T=2048, n_pos=64)
    assert not np.array_equal(host["K"], d["K"][0])          # a different random stream


def test_device_layers_regenerate_and_share_host_weights():
    a, b = _device_layer(layer=2), _device_layer(layer=2)
    assert all(np.array_equal(a[k], b[k]) for k in a)
    c = _device_layer(layer=3)
    assert not np.array_equal(a["K"], c["K"])
    assert not np.array_equal(a["K"][0], a["K"][1])           # heads differ
    idx = synth.make_indexer(W, 2, 1)
    assert all(np.array_equal(a[f][1], idx[f]) for f in idx)
    assert np.array_equal(a["X"], synth.make_layer_activations(W, 2, n_pos=64))
