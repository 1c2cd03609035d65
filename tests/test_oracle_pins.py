"""Pins of the fp64 CPU oracle to things other than itself.

Every check here compares the oracle with a library routine on a special case,
a closed form, an invariant the paper states, or brute force on tiny inputs.
The paper prints no worked numeric example, so no value is copied from it.
"""

import itertools
import math

import numpy as np
import pytest
import scipy.stats
import torch

import oracle
from paper_2608_08878_gb300 import synth


def bits(x):
    return synth.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def widen(b):
    return synth.bf16_bits_to_f32(b).astype(np.float64)


def rand_bits(rng, *shape, scale=1.0):
    return bits(rng.standard_normal(shape).astype(np.float32) * np.float32(scale))


def sdpa_gqa(q_bits, k_bits, v_bits):
    """torch's scaled_dot_product_attention in fp64 for one KV head's query group."""
    q = torch.from_numpy(widen(q_bits))[None, :, None, :]          # [1, G, 1, d]
    G = q.shape[1]
    k = torch.from_numpy(widen(k_bits))[None, None].expand(1, G, -1, -1)
    v = torch.from_numpy(widen(v_bits))[None, None].expand(1, G, -1, -1)
    o = torch.nn.functional.scaled_dot_product_attention(q, k, v)
    return o[0, :, 0, :].numpy()


def softmax_rows(q_bits, k_bits):
    q = torch.from_numpy(widen(q_bits))
    k = torch.from_numpy(widen(k_bits))
    return torch.softmax(q @ k.T / math.sqrt(q.shape[1]), dim=-1).numpy()  # [G][n]


# --------------------------------------------------------------------------
# Attention and entropy
# --------------------------------------------------------------------------

@pytest.mark.parametrize("n,d,G", [(1, 64, 2), (37, 64, 4), (300, 128, 4)])
def test_attention_equals_torch_sdpa(n, d, G):
    rng = np.random.default_rng(n + d)
    q, k, v = rand_bits(rng, G, d), rand_bits(rng, n, d, scale=2.0), rand_bits(rng, n, d)
    o, Hq = oracle.attend(q, k, v)
    np.testing.assert_allclose(o, sdpa_gqa(q, k, v), rtol=1e-12, atol=1e-12)
    a = softmax_rows(q, k)
    np.testing.assert_allclose(a.sum(-1), 1.0, rtol=1e-12)
    np.testing.assert_allclose(Hq, [scipy.stats.entropy(a[h]) for h in range(G)], rtol=1e-10, atol=1e-12)
    assert np.all(Hq >= -1e-12) and np.all(Hq <= math.log(n) + 1e-9)


def test_entropy_uniform_and_one_hot():
    d, n = 64, 50
    q = bits(np.ones((2, d)))
    k = bits(np.zeros((n, d)))
    v = bits(np.random.default_rng(0).standard_normal((n, d)))
    _, Hq = oracle.attend(q, k, v)
    np.testing.assert_allclose(Hq, math.log(n), rtol=1e-13)
    k2 = np.zeros((n, d), dtype=np.float32)
    k2[7] = 8.0  # one key far along q: its logit is 64 above the rest
    o, Hq2 = oracle.attend(q, bits(k2), v)
    assert np.all(Hq2 < 1e-20)
    np.testing.assert_allclose(o[0], widen(v[7]), rtol=1e-20, atol=1e-20)
    # logit 800 above the rest: the other weights underflow to exactly 0 in
    # fp64, and their terms 0 ln 0 count as 0 (the limit), so H is exactly 0
    k3 = np.zeros((n, d), dtype=np.float32)
    k3[7] = 100.0
    a3 = softmax_rows(q, bits(k3))
    assert np.count_nonzero(a3[0]) == 1
    _, Hq3 = oracle.attend(q, bits(k3), v)
    np.testing.assert_array_equal(Hq3, [scipy.stats.entropy(a3[h]) for h in range(2)])
    np.testing.assert_array_equal(Hq3, 0.0)


# --------------------------------------------------------------------------
# Step: features against library routines, closed forms and brute force
# --------------------------------------------------------------------------

def _mlp(hidden=16, layernorm=1, seed=3):
    return synth.policy_weights(seed, hidden), hidden, layernorm


def test_step_features_against_libraries():
    rng = np.random.default_rng(5)
    d, G, T = 32, 4, 40
    row = oracle.OracleRow(d, G, window=64, alpha_mode=0, capacity=64)
    kp, vp = rand_bits(rng, T, d), rand_bits(rng, T, d)
    row.append(kp, vp)
    q, kn, vn = rand_bits(rng, G, d), rand_bits(rng, d), rand_bits(rng, d)
    mlp, H, ln = _mlp()
    r = row.step(q, kn, vn, mlp, H, ln)
    K = np.concatenate([kp, kn[None]])
    V = np.concatenate([vp, vn[None]])
    a = softmax_rows(q, K)                                  # [G][n]
    at = torch.from_numpy(a)
    np.testing.assert_allclose(r["o"], sdpa_gqa(q, K, V), rtol=1e-12, atol=1e-12)
    f = r["feat"]
    np.testing.assert_allclose(f[:, 0], at.mean(0).numpy(), rtol=1e-12)                    # alpha
    np.testing.assert_allclose(f[:, 1], np.linalg.norm(widen(V), axis=1), rtol=1e-13)     # |v|
    np.testing.assert_allclose(f[:, 2], at.var(0, unbiased=False).numpy(), rtol=1e-9, atol=1e-20)
    # first step: the window holds one query step -> H_i = sum_h a_h H_h / sum_h a_h
    Hq = np.array([scipy.stats.entropy(a[h]) for h in range(G)])
    np.testing.assert_allclose(r["Hq"], Hq, rtol=1e-10)
    np.testing.assert_allclose(f[:, 3], (a * Hq[:, None]).sum(0) / a.sum(0), rtol=1e-10)
    np.testing.assert_allclose(f[:, 4], np.arange(T + 1) / T, rtol=1e-15)                   # pos
    np.testing.assert_array_equal(r["pos"], np.arange(T + 1))


def test_step_after_eviction_against_libraries():
    """A step after an eviction that removed tokens from the middle of the row:
    the survivors are a set the test picks (through the scores it passes), so
    every expected value is computed here from the test's own key/value arrays,
    never from the oracle's bookkeeping. Attention runs over the survivors plus
    the new token; pos_i divides the absolute position (tokens seen) by the
    newest one; with w = 2 the window sums pool the step before the eviction
    (over all T + 1 tokens) and this one, matched by position."""
    rng = np.random.default_rng(17)
    d, G, T = 32, 4, 30
    row = oracle.OracleRow(d, G, window=2, alpha_mode=0, capacity=64)
    kp, vp = rand_bits(rng, T, d), rand_bits(rng, T, d)
    row.append(kp, vp)
    mlp, H, ln = _mlp()
    q1, k1, v1 = rand_bits(rng, G, d), rand_bits(rng, d), rand_bits(rng, d)
    row.step(q1, k1, v1, mlp, H, ln)
    K1, V1 = np.concatenate([kp, k1[None]]), np.concatenate([vp, v1[None]])   # positions 0..T
    keep = np.sort(rng.choice(T + 1, size=11, replace=False))
    scores = np.full(T + 1, -1.0, dtype=np.float32)
    scores[keep] = 1.0 + np.arange(keep.size, dtype=np.float32)
    assert row.evict(keep.size, scores) == keep.size
    q2, k2, v2 = rand_bits(rng, G, d), rand_bits(rng, d), rand_bits(rng, d)
    r = row.step(q2, k2, v2, mlp, H, ln)
    pos = np.append(keep, T + 1)
    np.testing.assert_array_equal(r["pos"], pos)
    K2, V2 = np.concatenate([K1[keep], k2[None]]), np.concatenate([V1[keep], v2[None]])
    np.testing.assert_allclose(r["o"], sdpa_gqa(q2, K2, V2), rtol=1e-12, atol=1e-12)
    a1, a2 = softmax_rows(q1, K1), softmax_rows(q2, K2)                      # [G][T+1], [G][n]
    H1 = np.array([scipy.stats.entropy(a1[h]) for h in range(G)])
    H2 = np.array([scipy.stats.entropy(a2[h]) for h in range(G)])
    f = r["feat"]
    at = torch.from_numpy(a2)
    np.testing.assert_allclose(f[:, 0], at.mean(0).numpy(), rtol=1e-12)                    # alpha
    np.testing.assert_allclose(f[:, 1], np.linalg.norm(widen(V2), axis=1), rtol=1e-13)    # |v|
    np.testing.assert_allclose(f[:, 2], at.var(0, unbiased=False).numpy(), rtol=1e-9, atol=1e-20)
    Z = a2.sum(0)
    S = (a2 * H2[:, None]).sum(0)
    Z[:-1] += a1[:, keep].sum(0)                                # the survivors were attended before
    S[:-1] += (a1[:, keep] * H1[:, None]).sum(0)
    np.testing.assert_allclose(f[:, 3], S / Z, rtol=1e-10)                                  # H_i
    np.testing.assert_allclose(f[:, 4], pos / (T + 1), rtol=1e-15)                           # pos


def test_mlp_equals_torch_sequential():
    rng = np.random.default_rng(9)
    x = rng.standard_normal((200, 5)) * np.array([0.1, 10.0, 0.01, 3.0, 1.0])
    for hidden, layernorm in [(128, 1), (64, 0), (7, 1)]:
        blob = synth.policy_weights(11, hidden)
        # blob: [W1 5H | b1 H | gamma H | beta H | w2 H | b2]; give LayerNorm a
        # non-trivial gain and shift so both are exercised.
        blob[6 * hidden:7 * hidden] = 1.0 + 0.1 * np.arange(hidden, dtype=np.float32)
        blob[7 * hidden:8 * hidden] = (0.1 * rng.standard_normal(hidden)).astype(np.float32)
        W1 = blob[:5 * hidden].reshape(hidden, 5)
        b1 = blob[5 * hidden:6 * hidden]
        gamma = blob[6 * hidden:7 * hidden]
        beta = blob[7 * hidden:8 * hidden]
        w2 = blob[8 * hidden:9 * hidden]
        b2 = blob[9 * hidden]
        lin1 = torch.nn.Linear(5, hidden).double()
        lin2 = torch.nn.Linear(hidden, 1).double()
        with torch.no_grad():
            lin1.weight.copy_(torch.from_numpy(W1.astype(np.float64)))
            lin1.bias.copy_(torch.from_numpy(b1.astype(np.float64)))
            lin2.weight.copy_(torch.from_numpy(w2.astype(np.float64))[None])
            lin2.bias.fill_(float(b2))
        layers = [lin1]
        if layernorm:
            lnm = torch.nn.LayerNorm(hidden, eps=1e-5).double()
            with torch.no_grad():
                lnm.weight.copy_(torch.from_numpy(gamma.astype(np.float64)))
                lnm.bias.copy_(torch.from_numpy(beta.astype(np.float64)))
            layers.append(lnm)
        layers += [torch.nn.ReLU(), lin2]
        ref = torch.nn.Sequential(*layers)(torch.from_numpy(x)).detach().numpy()[:, 0]
        np.testing.assert_allclose(oracle.policy(x, blob, hidden, layernorm), ref, rtol=1e-12, atol=1e-12)


def test_uniform_keys_closed_forms():
    """All keys equal: every query attends uniformly, so a = 1/n, sigma = 0,
    H_q = ln n and (with a constant cache size) H_i = ln n for every token;
    cumulative alpha is (steps since insertion) / n."""
    d, G, B, T = 16, 2, 9, 20
    kc = bits(np.full((1, d), 0.5))
    rng = np.random.default_rng(1)
    mlp, H, ln = _mlp(8, 1)
    for mode in (0, 1):
        row = oracle.OracleRow(d, G, window=4, alpha_mode=mode, capacity=T + 1)
        row.append(np.repeat(kc, T, 0), rand_bits(rng, T, d))
        inserted = {p: 0 for p in range(T)}
        for step in range(10):
            r = row.step(rand_bits(rng, G, d), kc[0], rand_bits(rng, d), mlp, H, ln)
            n = len(r["pos"])
            inserted[int(r["pos"][-1])] = step
            np.testing.assert_allclose(r["Hq"], math.log(n), rtol=1e-13)
            assert np.all(r["feat"][:, 2] == 0.0)
            if step >= 4:  # the cache held B + 1 tokens at every step of the window
                np.testing.assert_allclose(r["feat"][:, 3], math.log(B + 1), rtol=1e-12)
            if mode == 0:
                np.testing.assert_allclose(r["feat"][:, 0], 1.0 / n, rtol=1e-13)
            elif step >= 1:
                want = [(step - max(inserted[int(p)], 1) + 1) / (B + 1) + (1.0 / (T + 1) if inserted[int(p)] == 0 else 0.0)
                        for p in r["pos"]]
                np.testing.assert_allclose(r["feat"][:, 0], want, rtol=1e-12)
            row.evict(B)


def _bruteforce_run(alpha_mode, w, steps, seed):
    rng = np.random.default_rng(seed)
    d, G, T, B = 8, 2, 6, 5
    mlp, H, ln = _mlp(8, 1)
    row = oracle.OracleRow(d, G, window=w, alpha_mode=alpha_mode, capacity=T + steps + 1)
    kp, vp = rand_bits(rng, T, d), rand_bits(rng, T, d)
    row.append(kp, vp)
    store_k = {p: kp[p] for p in range(T)}
    history = []  # per step: (dict pos -> a [G], H [G])
    for step in range(steps):
        q, kn, vn = rand_bits(rng, G, d, scale=1.5), rand_bits(rng, d), rand_bits(rng, d)
        r = row.step(q, kn, vn, mlp, H, ln)
        pos = r["pos"]
        store_k[int(pos[-1])] = kn
        K = np.stack([store_k[int(p)] for p in pos])
        a = softmax_rows(q, K)
        Hq = np.array([scipy.stats.entropy(a[h]) for h in range(G)])
        history.append(({int(p): a[:, i] for i, p in enumerate(pos)}, Hq))
        S_w, Z_w, acc = row.window_sums()
        S_p, Z_p = row.window_sums_prior()
        newest = history[-1][0]
        for i, p in enumerate(pos):
            np.testing.assert_allclose(Z_p[i] + newest[int(p)].sum(), Z_w[i], rtol=1e-12)
            np.testing.assert_allclose(S_p[i] + (newest[int(p)] * history[-1][1]).sum(), S_w[i], rtol=1e-12)
            Z = S = 0.0
            for amap, Hh in history[-w:]:
                if int(p) in amap:
                    Z += amap[int(p)].sum()
                    S += (amap[int(p)] * Hh).sum()
            np.testing.assert_allclose(Z_w[i], Z, rtol=1e-12)
            np.testing.assert_allclose(S_w[i], S, rtol=1e-12)
            np.testing.assert_allclose(r["feat"][i, 3], S / Z, rtol=1e-12)
            if alpha_mode == 1:
                cum = sum(amap[int(p)].mean() for amap, _ in history if int(p) in amap)
                np.testing.assert_allclose(r["feat"][i, 0], cum, rtol=1e-12)
        row.evict(B)
    return row


@pytest.mark.parametrize("w,alpha_mode", [(1, 0), (3, 0), (3, 1), (64, 0)])
def test_window_sums_brute_force(w, alpha_mode):
    _bruteforce_run(alpha_mode, w, steps=12, seed=w + 10 * alpha_mode)


# --------------------------------------------------------------------------
# Top-B selection and pruning
# --------------------------------------------------------------------------

def _lexsort_keep(scores, pos, B):
    s = np.asarray(scores, dtype=np.float64)
    nan = np.isnan(s)
    key = np.where(nan, 0.0, -s)  # descending score; -0 and +0 compare equal
    order = np.lexsort((pos, key, nan))
    return set(int(pos[i]) for i in order[:B])


def _row_with_n(n, d=4, G=1):
    rng = np.random.default_rng(n)
    row = oracle.OracleRow(d, G, window=4, alpha_mode=0, capacity=n + 1)
    row.append(rand_bits(rng, n, d), rand_bits(rng, n, d))
    return row


def test_evict_matches_lexsort_with_ties_zeros_and_nan():
    rng = np.random.default_rng(2)
    for n, B in [(1, 1), (10, 3), (64, 17), (100, 100), (100, 150)]:
        scores = rng.integers(-3, 4, n).astype(np.float32)  # many ties
        scores[rng.random(n) < 0.1] = -0.0
        scores[rng.random(n) < 0.05] = np.nan
        row = _row_with_n(n)
        pos = row.positions()
        want = _lexsort_keep(scores, pos, B)
        assert row.evict(B, scores) == min(n, B)
        assert set(row.positions().tolist()) == want
        assert np.all(np.diff(row.positions()) > 0)


def test_evict_brute_force_subsets():
    """The kept set is the B-subset whose ranking keys (score, -position) sort
    highest, found by enumerating every subset."""
    rng = np.random.default_rng(4)
    for trial in range(30):
        n = int(rng.integers(1, 8))
        B = int(rng.integers(1, n + 1))
        scores = rng.integers(-2, 3, n).astype(np.float32)
        row = _row_with_n(n)
        pos = row.positions()
        best = None
        for sub in itertools.combinations(range(n), B):
            key = sorted(((float(scores[i]), -int(pos[i])) for i in sub), reverse=True)
            if best is None or key > best[0]:
                best = (key, set(int(pos[i]) for i in sub))
        row.evict(B, scores)
        assert set(row.positions().tolist()) == best[1]


def test_prune_keeps_bytes_and_budget_invariants():
    wl = synth.TINY
    L, b, g = 0, 0, 1
    kp, vp = synth.prompt_row(wl, L, b, g)
    row = oracle.OracleRow(wl.head_dim, wl.group, wl.window, 0, wl.capacity)
    row.append(kp, vp)
    src_k = {p: kp[p] for p in range(wl.prompt_len)}
    src_v = {p: vp[p] for p in range(wl.prompt_len)}
    mlp = synth.policy_weights(wl.policy_seed, wl.mlp_hidden)
    for step in range(wl.steps):
        q, kn, vn = synth.step_row(wl, step, L, b, g)
        n_before = len(row) + 1
        r = row.step(q, kn, vn, mlp, wl.mlp_hidden, wl.layernorm)
        newest = int(r["pos"][-1])
        src_k[newest], src_v[newest] = kn, vn
        assert newest == wl.prompt_len + step and len(r["pos"]) == n_before
        row.evict(wl.budget)
        assert len(row) == min(n_before, wl.budget)
        k, v = row.kv_bits()
        for i, p in enumerate(row.positions()):
            assert np.array_equal(k[i], src_k[int(p)]) and np.array_equal(v[i], src_v[int(p)])


def test_budget_at_least_n_is_full_cache_attention():
    rng = np.random.default_rng(8)
    d, G, T = 32, 4, 25
    mlp, H, ln = _mlp()
    row = oracle.OracleRow(d, G, 64, 0, T + 20)
    K, V = rand_bits(rng, T, d), rand_bits(rng, T, d)
    row.append(K, V)
    for step in range(10):
        q, kn, vn = rand_bits(rng, G, d), rand_bits(rng, d), rand_bits(rng, d)
        r = row.step(q, kn, vn, mlp, H, ln)
        K, V = np.concatenate([K, kn[None]]), np.concatenate([V, vn[None]])
        np.testing.assert_allclose(r["o"], sdpa_gqa(q, K, V), rtol=1e-12, atol=1e-12)
        assert row.evict(T + 20) == len(K)


def test_paper_eviction_error_bound():
    """Sec. 3.1 (Reward): |o - o_hat| <= 2 C eps, with C = max |v_i| and eps the
    full-cache attention mass on the evicted tokens, against an unpruned
    teacher row fed the same inputs."""
    wl = synth.TINY.with_(prompt_len=96, budget=24, steps=20)
    mlp = synth.policy_weights(0, wl.mlp_hidden)
    kp, vp = synth.prompt_row(wl, 0, 0, 0)
    teacher = oracle.OracleRow(wl.head_dim, wl.group, wl.window, 0, wl.prompt_len + wl.steps + 1)
    student = oracle.OracleRow(wl.head_dim, wl.group, wl.window, 0, wl.prompt_len + wl.steps + 1)
    teacher.append(kp, vp)
    student.append(kp, vp)
    K = kp
    for step in range(wl.steps):
        q, kn, vn = synth.step_row(wl, step, 0, 0, 0)
        rt = teacher.step(q, kn, vn, mlp, wl.mlp_hidden, wl.layernorm)
        rs = student.step(q, kn, vn, mlp, wl.mlp_hidden, wl.layernorm)
        K = np.concatenate([K, kn[None]])
        a = softmax_rows(q, K)
        kept = np.isin(rt["pos"], rs["pos"])
        eps = a[:, ~kept].sum(1)
        Vt = widen(teacher.kv_bits()[1])
        C = np.linalg.norm(Vt, axis=1).max()
        err = np.linalg.norm(rt["o"] - rs["o"], axis=1)
        assert np.all(err <= 2 * C * eps + 1e-12), (step, err, eps)
        if step > 0:
            assert np.all(eps > 0)
        student.evict(wl.budget)


def test_capacity_overflow_leaves_row_unchanged():
    row = _row_with_n(4)
    with pytest.raises(OverflowError):
        row.append(np.zeros((2, 4), np.uint16), np.zeros((2, 4), np.uint16))
    assert len(row) == 4


# --------------------------------------------------------------------------
# Heuristic scorers (H2O, StreamingLLM) on the same path
# --------------------------------------------------------------------------

def test_h2o_scores_are_cumulative_mass_brute_force():
    """H2O ranks by the attention mass a token received since it entered the
    cache: recomputed here from torch softmax over every step's cache."""
    rng = np.random.default_rng(21)
    d, G, T, steps, B = 16, 2, 30, 6, 24
    row = oracle.OracleRow(d, G, 4, 1, T + steps + 2)
    k0, v0 = rand_bits(rng, T, d), rand_bits(rng, T, d)
    row.append(k0, v0)
    keys = {p: k0[p] for p in range(T)}
    mass = {p: 0.0 for p in range(T)}
    blob = synth.policy_weights(3, 8)
    for s in range(steps):
        q, kn, vn = rand_bits(rng, G, d), rand_bits(rng, 1, d)[0], rand_bits(rng, 1, d)[0]
        row.step(q, kn, vn, blob, 8, 1)
        p_new = T + s
        keys[p_new] = kn
        mass[p_new] = 0.0
        pos = row.positions()
        a = softmax_rows(q, np.stack([keys[p] for p in pos]))  # [G][n]
        for i, p in enumerate(pos):
            mass[p] += a[:, i].mean()
        h = row.heuristic_scores(1)
        np.testing.assert_allclose(h, [mass[p] for p in pos], rtol=1e-12, atol=1e-15)
        # evict with the H2O scores: the kept set is the top-B by (mass desc, position asc)
        want = sorted(pos, key=lambda p: (-mass[p], p))[:B]
        row.evict(B, h.astype(np.float32))
        assert sorted(row.positions().tolist()) == sorted(want)
        for p in set(mass) - set(row.positions().tolist()):
            mass.pop(p)


@pytest.mark.parametrize("n_sinks", [0, 4])
def test_streamingllm_keeps_sinks_and_most_recent(n_sinks):
    """StreamingLLM keeps the first n_sinks positions and then the most recent
    tokens: after every eviction the cache is exactly that set."""
    rng = np.random.default_rng(22)
    d, G, T, B = 8, 2, 40, 16
    row = oracle.OracleRow(d, G, 4, 0, T + 20)
    row.append(rand_bits(rng, T, d), rand_bits(rng, T, d))
    blob = synth.policy_weights(3, 8)
    for s in range(10):
        row.step(rand_bits(rng, G, d), rand_bits(rng, 1, d)[0], rand_bits(rng, 1, d)[0], blob, 8, 1)
        h = row.heuristic_scores(2, n_sinks)
        row.evict(B, h.astype(np.float32))
        newest = T + s
        want = list(range(n_sinks)) + list(range(newest - (B - n_sinks) + 1, newest + 1))
        assert row.positions().tolist() == want


# --------------------------------------------------------------------------
# Training side (App. C): Plackett-Luce log-partition, Gumbel-top-B
# --------------------------------------------------------------------------

@pytest.mark.parametrize("L", [1, 2, 5, 9])
def test_pl_logz_brute_force_subsets(L):
    """log Z is the log-sum-exp over every size-B subset of the subset's score
    sum / tau: enumerated here for every B."""
    from scipy.special import logsumexp
    rng = np.random.default_rng(30 + L)
    s = rng.standard_normal(L) * 3.0
    for tau in (1.0, 0.5):
        for B in range(1, L + 1):
            sums = [sum(s[list(a)]) / tau for a in itertools.combinations(range(L), B)]
            assert oracle.pl_logz(s, B, tau) == pytest.approx(logsumexp(sums), rel=1e-12, abs=1e-12)


def test_pl_logz_closed_forms():
    """B = 1: log-sum-exp of s / tau; B = L: sum of s / tau; equal scores c:
    log C(L, B) + B c / tau."""
    from scipy.special import logsumexp
    rng = np.random.default_rng(31)
    s = rng.standard_normal(1000) * 4.0
    assert oracle.pl_logz(s, 1, 0.7) == pytest.approx(logsumexp(s / 0.7), rel=1e-12)
    assert oracle.pl_logz(s, 1000, 0.7) == pytest.approx(s.sum() / 0.7, rel=1e-12)
    c, L, B = 1.25, 1000, 300
    want = math.lgamma(L + 1) - math.lgamma(B + 1) - math.lgamma(L - B + 1) + B * c
    assert oracle.pl_logz(np.full(L, c), B, 1.0) == pytest.approx(want, rel=1e-12)


def test_gumbel_topb_matches_lexsort():
    """The kept set is the B largest fp32 perturbed scores (ties: lower index),
    with -0 equal to +0: against numpy's lexsort on the same fp32 values."""
    rng = np.random.default_rng(32)
    L, B, tau = 500, 123, np.float32(0.5)
    s = np.round(rng.standard_normal(L) * 4).astype(np.float32)   # many ties
    g = np.zeros(L, dtype=np.float32)
    g[::3] = np.round(rng.gumbel(size=len(g[::3]))).astype(np.float32)
    s[7], g[7], s[8], g[8] = np.float32(-0.0), np.float32(0.0), np.float32(0.0), np.float32(0.0)
    v = (s / tau + g).astype(np.float32)
    v[v == 0] = 0.0
    order = np.lexsort((np.arange(L), -v.astype(np.float64)))
    want = np.sort(order[:B])
    assert np.array_equal(oracle.gumbel_topb(s, g, B, float(tau)), want)


def _pl_without_replacement_subset_prob(x, a):
    """Probability that sequential Plackett-Luce draws without replacement
    (weights x) pick exactly the set a in its first |a| draws: the sum over
    the orderings of a of prod_j x_j / (weight not yet drawn)."""
    total, p = float(sum(x)), 0.0
    for perm in itertools.permutations(a):
        rem, q = total, 1.0
        for i in perm:
            q *= x[i] / rem
            rem -= x[i]
        p += q
    return p


def test_gumbel_topb_samples_plackett_luce():
    """Gumbel-top-B draws the B items of Plackett-Luce sampling without
    replacement: subset frequencies of 40000 seeded draws against those
    probabilities. For B = 1 this is exp(s_i / tau - log Z) (App. C); for
    1 < B < L the subset law differs from exp(sum_a s / tau - log Z) (see the
    design notes), which the second half checks is a real difference."""
    rng = np.random.default_rng(33)
    L, tau, N = 5, 1.0, 40000
    s = np.array([1.0, 0.2, -0.5, 0.7, -1.2], dtype=np.float32)
    x = np.exp(s.astype(np.float64) / tau)
    g = rng.gumbel(size=(N, L)).astype(np.float32)
    for B in (1, 2):
        logz = oracle.pl_logz(s.astype(np.float64), B, tau)
        counts = {}
        for n in range(N):
            a = tuple(oracle.gumbel_topb(s, g[n], B, tau).tolist())
            counts[a] = counts.get(a, 0) + 1
        for a in itertools.combinations(range(L), B):
            p = _pl_without_replacement_subset_prob(x, a)
            sd = math.sqrt(p * (1 - p) / N)
            assert abs(counts.get(a, 0) / N - p) < 5 * sd + 1e-4, (B, a, counts.get(a, 0) / N, p)
            p_paper = math.exp(float(s[list(a)].astype(np.float64).sum()) / tau - logz)
            if B == 1:
                assert p_paper == pytest.approx(p, rel=1e-12)
        if B == 2:
            a = (0, 3)
            assert abs(_pl_without_replacement_subset_prob(x, a) -
                       math.exp(float(s[list(a)].astype(np.float64).sum()) / tau - logz)) > 0.02


# --------------------------------------------------------------------------
# Global token mode (features over all heads and layers of a sequence)
# --------------------------------------------------------------------------

def test_global_mode_with_one_row_is_the_row_oracle():
    """A sequence of one row pools nothing: every step's features, scores,
    window sums and evictions equal the per-row oracle's."""
    rng = np.random.default_rng(40)
    d, G, T, w, cap = 16, 4, 60, 3, 80
    blob = synth.policy_weights(5, 32)
    row = oracle.OracleRow(d, G, w, 1, cap)
    seq = oracle.OracleSeq(1, d, G, w, 1, cap)
    k, v = rand_bits(rng, T, d), rand_bits(rng, T, d)
    row.append(k, v)
    seq.append(k[None], v[None])
    for s in range(8):
        q, kn, vn = rand_bits(rng, G, d), rand_bits(rng, 1, d)[0], rand_bits(rng, 1, d)[0]
        a = row.step(q, kn, vn, blob, 32, 1)
        b = seq.step(q[None], kn[None], vn[None], blob, 32, 1)
        np.testing.assert_allclose(b["o"][0], a["o"], rtol=0, atol=0)
        np.testing.assert_allclose(b["feat"], a["feat"], rtol=1e-13, atol=1e-15)
        np.testing.assert_allclose(b["score"], a["score"], rtol=1e-13, atol=1e-15)
        np.testing.assert_allclose(seq.window_sums_prior(), row.window_sums_prior(), rtol=1e-13, atol=1e-15)
        row.evict(50)
        seq.evict(50)
        assert np.array_equal(row.positions(), seq.positions())
        assert all(np.array_equal(x, y) for x, y in zip(row.kv_bits(), seq.kv_bits(0)))


@pytest.mark.parametrize("alpha_mode", [0, 1])
def test_global_mode_pooled_features_brute_force(alpha_mode):
    """alpha, sigma, |v|, H and pos of a 3-row sequence recomputed from torch
    softmax over every row's heads, stacked, over a 3-step window, and the
    window sums without the latest step; in alpha_mode 1 alpha is the pooled
    mass summed over the steps since the token's insertion. Every row pruned to
    the same survivors, which are the sequence's top-B."""
    rng = np.random.default_rng(41)
    R, d, G, T, w, B = 3, 16, 2, 25, 3, 20
    blob = synth.policy_weights(6, 32)
    seq = oracle.OracleSeq(R, d, G, w, alpha_mode, T + 10)
    acc = {}  # position -> pooled mass summed over the steps since insertion
    K = {r: list(rand_bits(rng, T, d)) for r in range(R)}
    V = {r: list(rand_bits(rng, T, d)) for r in range(R)}
    seq.append(np.stack([np.stack(K[r]) for r in range(R)]), np.stack([np.stack(V[r]) for r in range(R)]))
    pos = list(range(T))
    hist = []  # per step: {position: (sum a, sum a H)}
    for s in range(6):
        q = rand_bits(rng, R, G, d)
        kn, vn = rand_bits(rng, R, d), rand_bits(rng, R, d)
        for r in range(R):
            K[r].append(kn[r]); V[r].append(vn[r])
        pos.append(T + s)
        res = seq.step(q, kn, vn, blob, 32, 1)
        a = np.concatenate([softmax_rows(q[r], np.stack(K[r])) for r in range(R)])  # [R*G][n]
        Hh = np.array([scipy.stats.entropy(a[j]) for j in range(R * G)])
        hist.append({p: (a[:, i].sum(), (a[:, i] * Hh).sum()) for i, p in enumerate(pos)})
        hist = hist[-w:]
        vnorm = np.mean([np.linalg.norm(widen(np.stack(V[r])), axis=1) for r in range(R)], axis=0)
        S = np.array([sum(h[p][1] for h in hist if p in h) for p in pos])
        Z = np.array([sum(h[p][0] for h in hist if p in h) for p in pos])
        for i, p in enumerate(pos):
            acc[p] = acc.get(p, 0.0) + a[:, i].mean()
        alpha = np.array([acc[p] for p in pos]) if alpha_mode else a.mean(0)
        want = np.stack([alpha, vnorm, a.var(0), np.where(Z > 0, S / Z, 0.0),
                         np.array(pos) / max(pos[-1], 1)], axis=1)
        np.testing.assert_allclose(res["feat"], want, rtol=1e-11, atol=1e-14)
        Sp, Zp = seq.window_sums_prior()
        np.testing.assert_allclose(Sp, [sum(h[p][1] for h in hist[:-1] if p in h) for p in pos], rtol=1e-12,
                                   atol=1e-15)
        np.testing.assert_allclose(Zp, [sum(h[p][0] for h in hist[:-1] if p in h) for p in pos], rtol=1e-12,
                                   atol=1e-15)
        sc = res["score"].astype(np.float32)
        keep = np.sort(np.lexsort((np.array(pos), -sc.astype(np.float64)))[:B])
        seq.evict(B, sc)
        kept_pos = [pos[i] for i in keep]
        assert seq.positions().tolist() == kept_pos
        for r in range(R):
            K[r] = [K[r][i] for i in keep]
            V[r] = [V[r][i] for i in keep]
            kb, vb = seq.kv_bits(r)
            assert np.array_equal(kb, np.stack(K[r])) and np.array_equal(vb, np.stack(V[r]))
        pos = kept_pos


# --------------------------------------------------------------------------
# Invariants on random rows (property-based)
# --------------------------------------------------------------------------

def test_step_invariants_on_random_rows():
    """Invariants that hold for any input, checked on random small rows over
    several steps with evictions: each step's alpha sums to 1 (alpha_mode 0);
    sigma lies in [0, alpha (1 - alpha)] (the variance of values in [0, 1] with
    that mean, population form); H_i lies in [0, ln of the longest row the
    window saw]; pos_i in [0, 1]; every output coordinate lies within the value
    rows' range (a convex combination); cumulative alpha (mode 1) is
    non-negative and sums to at most the number of steps."""
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    @hyp.settings(max_examples=60, deadline=None)
    @hyp.given(n=st.integers(1, 160), G=st.sampled_from([1, 2, 4]), w=st.integers(1, 6), steps=st.integers(1, 7),
               alpha_mode=st.integers(0, 1), seed=st.integers(0, 2 ** 31 - 1), data=st.data())
    def run(n, G, w, steps, alpha_mode, seed, data):
        rng = np.random.default_rng(seed)
        d = 64
        B = data.draw(st.integers(1, n + steps))
        row = oracle.OracleRow(d, G, w, alpha_mode, n + steps + 1)
        k = rand_bits(rng, n, d, scale=2.0)
        v = rand_bits(rng, n, d)
        row.append(k, v)
        blob = synth.policy_weights(0, 32)
        longest = n
        for s in range(steps):
            q = rand_bits(rng, G, d, scale=1.5)
            kn, vn = rand_bits(rng, 1, d, scale=2.0)[0], rand_bits(rng, 1, d)[0]
            vrows = np.concatenate([widen(row.kv_bits()[1]), widen(vn)[None]], axis=0) if len(row) else widen(vn)[None]
            res = row.step(q, kn, vn, blob, 32, 1)
            m = len(res["pos"])
            longest = max(longest, m)
            alpha, sigma, H, pos = res["feat"][:, 0], res["feat"][:, 2], res["feat"][:, 3], res["feat"][:, 4]
            if alpha_mode == 0:
                assert abs(alpha.sum() - 1.0) < 1e-12
                assert np.all(sigma >= -1e-15) and np.all(sigma <= alpha * (1 - alpha) + 1e-12)
            else:
                assert np.all(alpha >= -1e-15) and alpha.sum() <= s + 1 + 1e-9
            assert np.all(H >= -1e-12) and np.all(H <= math.log(longest) + 1e-12)
            assert np.all(pos >= 0) and np.all(pos <= 1)
            lo, hi = vrows.min(axis=0), vrows.max(axis=0)
            assert np.all(res["o"] >= lo - 1e-12) and np.all(res["o"] <= hi + 1e-12)
            row.evict(B)

    run()


def test_global_mode_invariants_on_random_sequences():
    """The same invariants in the global token mode, where a token's alpha,
    sigma and H pool every (row, head) pair of the sequence: alpha sums to 1,
    sigma in [0, alpha (1 - alpha)], 0 <= H <= ln n, pos in [0, 1], |v| the
    mean of the rows' value norms, each row's output inside its value range."""
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    @hyp.settings(max_examples=30, deadline=None)
    @hyp.given(R=st.integers(1, 4), n=st.integers(1, 80), G=st.sampled_from([1, 2, 4]), w=st.integers(1, 4),
               steps=st.integers(1, 5), seed=st.integers(0, 2 ** 31 - 1), data=st.data())
    def run(R, n, G, w, steps, seed, data):
        rng = np.random.default_rng(seed)
        d = 64
        B = data.draw(st.integers(1, n + steps))
        seq = oracle.OracleSeq(R, d, G, w, 0, n + steps + 1)
        seq.append(rand_bits(rng, R, n, d, scale=2.0), rand_bits(rng, R, n, d))
        blob = synth.policy_weights(0, 32)
        longest = n
        for _ in range(steps):
            q = rand_bits(rng, R, G, d, scale=1.5)
            kn, vn = rand_bits(rng, R, d, scale=2.0), rand_bits(rng, R, d)
            vrows = [np.concatenate([widen(seq.kv_bits(r)[1]), widen(vn[r])[None]], axis=0) for r in range(R)]
            res = seq.step(q, kn, vn, blob, 32, 1)
            longest = max(longest, len(res["pos"]))
            alpha, vnorm, sigma, H, pos = (res["feat"][:, c] for c in range(5))
            assert abs(alpha.sum() - 1.0) < 1e-12
            assert np.all(sigma >= -1e-15) and np.all(sigma <= alpha * (1 - alpha) + 1e-12)
            assert np.all(H >= -1e-12) and np.all(H <= math.log(longest) + 1e-12)
            assert np.all(pos >= 0) and np.all(pos <= 1)
            np.testing.assert_allclose(vnorm, np.mean([np.linalg.norm(vr, axis=1) for vr in vrows], axis=0),
                                       rtol=1e-12)
            for r in range(R):
                lo, hi = vrows[r].min(axis=0), vrows[r].max(axis=0)
                assert np.all(res["o"][r] >= lo - 1e-12) and np.all(res["o"][r] <= hi + 1e-12)
            seq.evict(B)

    run()
