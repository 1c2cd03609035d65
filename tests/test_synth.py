"""The seeded input generator: published SplitMix64 outputs, bf16 rounding
against torch, and the statistics of the synthetic workloads."""

import numpy as np
import torch

from paper_2608_08878_gb300 import synth


def test_splitmix64_published_sequence():
    # First outputs of the SplitMix64 generator seeded with 0 (state advances by
    # the golden gamma before each output).
    want = [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    got = [synth.splitmix64_int((i * 0x9E3779B97F4A7C15) & synth.MASK64) for i in range(3)]
    assert got == want
    arr = synth.splitmix64(np.array([(i * 0x9E3779B97F4A7C15) & synth.MASK64 for i in range(3)], dtype=np.uint64))
    assert [int(x) for x in arr] == want


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 10,
                        np.array([0.0, -0.0, 1.0, 65504.0, 1e-30, -3.3895314e38], dtype=np.float32)])
    ours = synth.f32_to_bf16_bits(x)
    theirs = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(ours, theirs)
    np.testing.assert_array_equal(synth.bf16_bits_to_f32(ours), torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_normal_stream_statistics_and_exactness():
    z = synth.normal_f32(synth.mix(1, 2, 3), 200000)
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1.0) < 0.01
    # exact in fp32: every value is an integer multiple of 2^-16
    assert np.all((z * 65536.0) == np.round(z * 65536.0))
    np.testing.assert_array_equal(synth.normal_rows_f32([synth.mix(1, 2, 3)], 50)[0], z[:50])


def test_workload_structure():
    wl = synth.MISTRAL_1L
    k, v = synth.prompt_row(wl, 0, 0, 3)
    kf = synth.bf16_bits_to_f32(k)
    hs = synth.hot_set(wl, 0, 0, 3, np.arange(wl.prompt_len))
    frac = (hs >= 0).mean()
    assert 0.005 < frac < 0.015
    u = synth.direction(wl, 0, 0, 3)
    cos = (kf @ u) / (np.linalg.norm(kf, axis=1) * np.linalg.norm(u))
    assert cos[hs >= 0].mean() > 0.8 and abs(cos[hs < 0][wl.n_sinks:].mean()) < 0.05
    sink_norm = np.linalg.norm(kf[:wl.n_sinks], axis=1).mean()
    rest = np.linalg.norm(kf[wl.n_sinks:][hs[wl.n_sinks:] < 0], axis=1).mean()
    assert 3.5 < sink_norm / rest < 4.5
    q, kn, vn = synth.step_row(wl, 5, 0, 0, 3)
    assert q.shape == (wl.group, wl.head_dim) and kn.shape == (wl.head_dim,)
    # deterministic
    np.testing.assert_array_equal(synth.prompt_row(wl, 0, 0, 3, 100, 200)[0], k[100:200])


def test_policy_weights_ranges():
    for H in (64, 128):
        w = synth.policy_weights(0, H)
        assert w.shape == (synth.policy_blob_len(H),)
        assert np.all(np.abs(w[:6 * H]) <= 1 / np.sqrt(5))
        np.testing.assert_array_equal(w[6 * H:7 * H], 1.0)
        np.testing.assert_array_equal(w[7 * H:8 * H], 0.0)
        assert np.all(np.abs(w[8 * H:]) <= 1 / np.sqrt(H))
