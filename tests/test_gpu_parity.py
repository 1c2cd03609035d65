"""CUDA path (through the C ABI) against the fp64 oracle on the same seeded
inputs: attention output, per-head entropy, the five features, policy scores,
the retained sets (oracle fed the GPU's scores), compacted K/V bytes and the
window state. Small cases run every row; the full-size workloads run in the
benchmark's launch configuration and check a sample of rows."""

import numpy as np
import pytest

from paper_2608_08878_gb300 import synth

from harness import LockStep, SeqLockStep, check_attention

pytestmark = pytest.mark.gpu

ENGINES = [1, 2]  # split, fused (forced wherever the step fits it)


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_08878_gb300 import build
    build.build()
    import torch
    torch.cuda.init()


def _bits(t):
    import torch
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def test_device_generator_matches_host():
    from paper_2608_08878_gb300 import synth_device
    for wl in (synth.TINY, synth.MISTRAL_1L.with_(prompt_len=300), synth.AGGRESSIVE.with_(layers=2, batch=2)):
        k, v = synth_device.prompt(wl, 0, min(wl.prompt_len, 300))
        kb, vb = _bits(k), _bits(v)
        for r in (0, wl.rows - 1, wl.rows // 2):
            layer, b, g = wl.row_coords(r)
            hk, hv = synth.prompt_row(wl, layer, b, g, 0, min(wl.prompt_len, 300))
            assert np.array_equal(kb[layer, b, g], hk) and np.array_equal(vb[layer, b, g], hv)
        for step in (0, 17, 40):
            q, kn, vn = synth_device.step_inputs(wl, step)
            hq, hk, hv = synth.step_all(wl, step) if wl.rows <= 64 else (None, None, None)
            if hq is not None:
                assert np.array_equal(_bits(q), hq) and np.array_equal(_bits(kn), hk)
                assert np.array_equal(_bits(vn), hv)


@pytest.mark.parametrize("engine", ENGINES)
def test_tiny_all_rows(engine):
    wl = synth.TINY
    ls = LockStep(wl, range(wl.rows), engine=engine)
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()
    assert ls.stats["evicted"] == (wl.prompt_len + 1 - wl.budget) + (wl.steps - 1)


@pytest.mark.parametrize("engine", ENGINES)
@pytest.mark.parametrize("alpha_mode", [0, 1])
def test_window_departure(engine, alpha_mode):
    wl = synth.TINY.with_(window=4, steps=32, prompt_len=200, budget=60, alpha_mode=alpha_mode)
    ls = LockStep(wl, range(wl.rows), engine=engine)
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()


@pytest.mark.parametrize("engine", ENGINES)
@pytest.mark.parametrize("prompt_len,budget", [(0, 3), (1, 1), (126, 40), (129, 128), (300, 299)])
def test_ragged_lengths(engine, prompt_len, budget):
    wl = synth.TINY.with_(prompt_len=prompt_len, budget=budget, steps=6, window=3)
    ls = LockStep(wl, range(wl.rows), engine=engine, capacity=max(prompt_len, budget) + 8)
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()


@pytest.mark.parametrize("engine", ENGINES)
def test_budget_at_least_n_is_full_attention(engine):
    import torch
    wl = synth.MISTRAL_1L.with_(prompt_len=500, budget=600, steps=4)
    ls = LockStep(wl, [0, 5], engine=engine, capacity=700)
    ls.load_prompt()
    for s in range(wl.steps):
        out = ls.step()
        q, _, _ = ls._inputs(s)
        full = ls.cache.full_decode(q)
        torch.cuda.synchronize()
        assert torch.allclose(out, full, atol=2e-3, rtol=0), float((out - full).abs().max())
    assert ls.cache.length()[0] == 504


@pytest.mark.parametrize("engine", ENGINES)
def test_mistral_single_layer(engine):
    """The Mistral-7B single-layer workload as specified: all 8 rows, 8192-token
    prompt compressed to 2048, 128 decode steps each evicting one token (queries
    leave the 64-step window from step 64 on)."""
    wl = synth.MISTRAL_1L
    assert wl.steps == 128
    ls = LockStep(wl, range(wl.rows), engine=engine)
    ls.load_prompt()
    for s in range(wl.steps):
        ls.step(check=(s < 3 or s % 8 == 0 or s >= 124))
    assert ls.cache.length()[0] == wl.budget


@pytest.mark.parametrize("engine", ENGINES)
def test_step_equals_decode_then_evict(engine):
    """dc_step (one kernel on the fused engine) leaves the cache and output
    bit-identical to dc_decode_step followed by dc_evict."""
    import torch
    from paper_2608_08878_gb300 import dc
    wl = synth.MISTRAL_1L.with_(prompt_len=700, budget=256, window=5)
    a, b = LockStep(wl, [], engine=engine), LockStep(wl, [], engine=engine)
    a.load_prompt()
    b.load_prompt()
    for s in range(12):
        q, kn, vn = a._inputs(s)
        budget = 200 if s == 6 else 0  # one step with a smaller budget: many evictions
        oa = a.cache.step(q, kn, vn, budget=budget)
        ob = b.cache.decode_step(q, kn, vn)
        b.cache.evict(budget)
        torch.cuda.synchronize()
        assert torch.equal(oa, ob), s
        assert a.cache.length() == b.cache.length()
        n = a.cache.length()[0]
        for which in (dc.BUF_K, dc.BUF_V, dc.BUF_POS, dc.BUF_S, dc.BUF_Z):
            assert torch.equal(a.cache.buffer(which)[:, :n], b.cache.buffer(which)[:, :n]), (s, which)


def _tail_workload(**kw):
    """Mistral-7B head shapes with a few more rows than SMs, so that the fused
    grid's last wave is partly filled and its rows are split in halves."""
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    batch = sms // 8 + 1
    wl = synth.MISTRAL_1L.with_(batch=batch, **kw)
    assert 0 < wl.rows - sms <= sms // 2
    return wl, sms


def test_tail_split_rows_match_oracle():
    """Half rows (two CTAs per row, statistics and output exchanged) against
    the oracle, across the window's departures. Rows of 3001 tokens (24
    tiles): longer than row pairs take."""
    wl, sms = _tail_workload(prompt_len=4000, budget=3000, steps=70)
    ls = LockStep(wl, [0, sms - 1, sms, sms + 3, wl.rows - 1], engine=2)
    ls.load_prompt()
    for s in range(wl.steps):
        ls.step(check=(s < 3 or s % 16 == 0 or s >= 66))


def test_tail_split_step_equals_decode_then_evict():
    """With half rows, dc_step's in-kernel eviction (candidates exchanged
    between the halves) leaves the cache bit-identical to dc_decode_step and
    dc_evict; the output agrees with whole-row CTAs to rounding."""
    import torch
    from paper_2608_08878_gb300 import dc
    wl, _ = _tail_workload(prompt_len=3500, budget=2800, window=6)  # 22 tiles: no row pairs
    a, b = LockStep(wl, [], engine=2), LockStep(wl, [], engine=2)
    c = LockStep(wl, [], engine=2, tail_split=False)
    for x in (a, b, c):
        x.load_prompt()
    for s in range(10):
        q, kn, vn = a._inputs(s)
        oa = a.cache.step(q, kn, vn)
        ob = b.cache.decode_step(q, kn, vn)
        b.cache.evict()
        oc = c.cache.step(q, kn, vn)
        a.cache.sync()
        b.cache.sync()
        c.cache.sync()
        assert torch.equal(oa, ob), s
        assert a.cache.length() == b.cache.length()
        n = a.cache.length()[0]
        for which in (dc.BUF_K, dc.BUF_V, dc.BUF_POS, dc.BUF_S, dc.BUF_Z, dc.BUF_VNORM):
            assert torch.equal(a.cache.buffer(which)[:, :n], b.cache.buffer(which)[:, :n]), (s, which)
        if s == 0:  # before the two caches' evictions could part on near-ties
            err = float((oa - oc).abs().max())
            assert err <= 1e-4, err


@pytest.mark.parametrize("group,head_dim,steps,alpha_mode", [(4, 128, 70, 0), (2, 128, 12, 1), (1, 64, 12, 0)])
def test_row_pairs_match_oracle(group, head_dim, steps, alpha_mode):
    """Row pairs (more rows than SMs, rows of at most 21 tiles: each
    warpgroup of a CTA does one row of the pair, their tiles alternating in
    the stage ring) against the oracle: both rows of the first and last
    pairs and of pairs on either side of the first wave, prompt compression
    (many evictions, one radix select per warpgroup) and steady steps across
    the window's departures."""
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    # four rows per SM: two pairs per CTA
    wl = synth.MISTRAL_1L.with_(batch=sms // 2, prompt_len=1500, budget=600, steps=steps, q_heads=8 * group,
                                head_dim=head_dim, alpha_mode=alpha_mode)
    assert wl.rows == 4 * sms
    ls = LockStep(wl, [0, 1, 2 * sms - 2, 2 * sms - 1, wl.rows - 2, wl.rows - 1], engine=2)
    assert ls.cache.engine(wl.prompt_len + 1) == "fused-pairs" and ls.cache.engine(wl.budget + 1) == "fused-pairs"
    ls.load_prompt()
    for s in range(wl.steps):
        ls.step(check=(s < 3 or s % 16 == 0 or s >= wl.steps - 4))
    assert ls.cache.length()[0] == wl.budget


def test_row_pairs_step_equals_decode_then_evict():
    """On row pairs, dc_step's in-kernel eviction (a radix select per
    warpgroup on the prompt compression, then one eviction per step) leaves
    the cache bit-identical to dc_decode_step and dc_evict, with the same
    output."""
    import torch
    from paper_2608_08878_gb300 import dc
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    wl = synth.MISTRAL_1L.with_(batch=sms // 2, prompt_len=2000, budget=500, window=6)
    a, b = LockStep(wl, [], engine=2), LockStep(wl, [], engine=2)
    assert a.cache.engine(wl.prompt_len + 1) == "fused-pairs" and a.cache.engine(wl.budget + 1) == "fused-pairs"
    for x in (a, b):
        x.load_prompt()
    for s in range(10):
        q, kn, vn = a._inputs(s)
        oa = a.cache.step(q, kn, vn)
        ob = b.cache.decode_step(q, kn, vn)
        b.cache.evict()
        a.cache.sync()
        b.cache.sync()
        assert torch.equal(oa, ob), s
        assert a.cache.length() == b.cache.length()
        n = a.cache.length()[0]
        for which in (dc.BUF_K, dc.BUF_V, dc.BUF_POS, dc.BUF_S, dc.BUF_Z, dc.BUF_VNORM):
            assert torch.equal(a.cache.buffer(which)[:, :n], b.cache.buffer(which)[:, :n]), (s, which)


@pytest.mark.parametrize("prompt_len,budget", [(12000, 10000), (16000, 12000)])
def test_fused_long_rows(prompt_len, budget):
    """Rows longer than the fused kernel keeps on chip (8704 tokens with four
    query heads per KV head): later tiles' logits go through HBM, and past
    10240 tokens the scores too. Prompt compression (many evictions) and
    steady steps, all 8 rows against the oracle."""
    wl = synth.MISTRAL_1L.with_(prompt_len=prompt_len, budget=budget, steps=4)
    ls = LockStep(wl, range(wl.rows), engine=2)
    assert ls.cache.engine() == "fused"
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()
    assert ls.cache.length()[0] == budget


@pytest.mark.parametrize("engine", ENGINES)
@pytest.mark.parametrize("scorer", [1, 2])
def test_heuristic_scorers(engine, scorer):
    """H2O (cumulative attention mass) and StreamingLLM (sinks + recent) on the
    same attention/top-k/compaction path, all rows, past the window; then
    dc_step bit-identical to dc_decode_step + dc_evict with that scorer."""
    import torch
    from paper_2608_08878_gb300 import dc
    wl = synth.MISTRAL_1L.with_(prompt_len=900, budget=300, steps=70)
    ls = LockStep(wl, range(wl.rows), engine=engine, scorer=scorer)
    ls.load_prompt()
    for s in range(wl.steps):
        ls.step(check=(s < 3 or s % 16 == 0 or s >= 66))
    wl2 = wl.with_(window=5)
    a = LockStep(wl2, [], engine=engine, scorer=scorer)
    b = LockStep(wl2, [], engine=engine, scorer=scorer)
    a.load_prompt()
    b.load_prompt()
    for s in range(8):
        q, kn, vn = a._inputs(s)
        oa = a.cache.step(q, kn, vn)
        ob = b.cache.decode_step(q, kn, vn)
        b.cache.evict()
        torch.cuda.synchronize()
        assert torch.equal(oa, ob), s
        n = a.cache.length()[0]
        for which in (dc.BUF_K, dc.BUF_POS, dc.BUF_S, dc.BUF_Z):
            assert torch.equal(a.cache.buffer(which)[:, :n], b.cache.buffer(which)[:, :n]), (s, which)


@pytest.mark.parametrize("n_sinks", [10000, 5000, 512])
def test_many_evictions_with_tied_scores(n_sinks):
    """The eviction kernel's select on a 12001-token row with budget 1024,
    StreamingLLM scores (the first n_sinks positions tie at the top, the rest
    are distinct): 10000 tied keys (more than the select lists in shared
    memory, so it takes its radix passes over the whole row), 5000 tied keys
    (listed, the cut among them by position), and 512 (the threshold among the
    distinct scores, survivors moved into the holes). Against the oracle fed
    the GPU's scores, then two steps with one eviction each."""
    wl = synth.MISTRAL_1L.with_(prompt_len=12000, budget=1024, steps=3)
    ls = LockStep(wl, [0, 5], engine=2, scorer=2, n_sinks=n_sinks)
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()
    assert ls.cache.length()[0] == 1024


@pytest.mark.parametrize("engine", ENGINES)
@pytest.mark.parametrize("basis", [0, 1])
def test_dynamic_budget(engine, basis):
    """B_t = max(floor(r L_t), B_min) with L_t the tokens seen (basis 0: the
    cache grows with the sequence) or the cached tokens (basis 1: it shrinks to
    B_min); every step checked against the oracle with that budget."""
    wl = synth.MISTRAL_1L.with_(prompt_len=700, budget=600, steps=12)
    cap = wl.prompt_len + wl.steps + 8
    ls = LockStep(wl, range(wl.rows), engine=engine, capacity=cap, budget_ratio=0.25, budget_min=32,
                  budget_basis=basis)
    ls.load_prompt()
    lengths = []
    for _ in range(wl.steps):
        ls.step()
        lengths.append(ls.cache.length()[0])
    if basis == 0:
        assert lengths[-1] == (wl.prompt_len + wl.steps) // 4
    else:
        assert lengths[:4] == [175, 44, 32, 32] and lengths[-1] == 32


@pytest.mark.parametrize("engine", ENGINES)
def test_per_row_budgets_head_level_hybrid(engine):
    """Per-row budgets (head-level hybrid, Sec. 5): 2 of 8 KV heads keep the
    full cache, the rest share a 25% overall budget; every row against the
    oracle with its own budget, through prompt compression and steady steps;
    then dc_step (the fused kernel's in-kernel selection per row) against
    dc_decode_step + dc_evict."""
    import torch
    from paper_2608_08878_gb300 import dc
    wl = synth.MISTRAL_1L.with_(prompt_len=1200, budget=300, steps=20)
    cap = wl.prompt_len + wl.steps + 8
    budgets = dc.head_level_hybrid_budgets(wl.rows, cap, full_rows=[1, 6], overall_ratio=0.25)
    assert budgets[1] == cap and budgets[6] == cap and budgets[0] < cap
    a = LockStep(wl, [], engine=engine, capacity=cap, row_budgets=budgets)
    b = LockStep(wl, [], engine=engine, capacity=cap, row_budgets=budgets)
    a.load_prompt()
    b.load_prompt()
    for s in range(6):
        q, kn, vn = a._inputs(s)
        oa = a.cache.step(q, kn, vn)
        ob = b.cache.decode_step(q, kn, vn)
        b.cache.evict()
        torch.cuda.synchronize()
        assert torch.equal(oa, ob), s
        assert np.array_equal(a.cache.row_lengths(), b.cache.row_lengths())
        for r in range(wl.rows):
            n = int(a.cache.row_lengths()[r])
            for which in (dc.BUF_K, dc.BUF_POS, dc.BUF_S, dc.BUF_Z):
                assert torch.equal(a.cache.buffer(which, r, 1)[:, :n], b.cache.buffer(which, r, 1)[:, :n]), (s, r)
    ls = LockStep(wl, range(wl.rows), engine=engine, capacity=cap, row_budgets=budgets)
    assert ls.cache.engine() == ("fused" if engine == 2 else "split")
    ls.load_prompt()
    for s in range(wl.steps):
        ls.step(check=(s < 3 or s >= 17))
    lens = ls.cache.row_lengths()
    assert lens[1] == wl.prompt_len + wl.steps and lens[0] == budgets[0]
    with pytest.raises(dc.DCError):
        ls.cache.full_decode(ls._inputs(0)[0])
    with pytest.raises(dc.DCError):
        ls.cache.set_row_budgets(None)  # rows differ in length


def test_engine_choice():
    from paper_2608_08878_gb300 import dc
    big = dc.DistillCache(32, 8, 128, 200, 100, batch=1)
    # 256 rows on the GPU's SMs: short rows go in pairs, long ones one per CTA
    assert big.engine() == "fused-pairs" and big.engine(400) == "fused-pairs"
    assert big.engine(3000) == "fused" and big.engine(20000) == "fused"
    # two rows: short ones on the fused kernel, long ones spread by the split engine
    small = dc.DistillCache(1, 2, 64, 30000, 100, q_heads=4)
    assert small.engine() == "fused" and small.engine(20000) == "split"
    forced = dc.DistillCache(1, 2, 64, 200, 100, q_heads=4, engine=2)
    assert forced.engine() == "fused"
    assert dc.DistillCache(1, 2, 64, 200, 100, q_heads=16, engine=2).engine() == "fused"  # group 8
    # a policy wider than the fused kernel's 128 hidden units stays on the split engine
    assert dc.DistillCache(1, 2, 64, 200, 100, q_heads=4, mlp_hidden=256, engine=2).engine() == "split"


def test_full_decode_matches_oracle():
    import torch
    import oracle
    from paper_2608_08878_gb300 import dc
    wl = synth.MISTRAL_1L.with_(prompt_len=3000)
    k, v = synth.prompt_all(wl)
    q, _, _ = synth.step_all(wl, 0)
    f = lambda a: torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).cuda()
    cache = dc.DistillCache(1, 8, 128, 3001, 100)
    cache.append(f(k), f(v))
    out = cache.full_decode(f(q)).cpu().numpy()
    for g in range(8):
        o, _ = oracle.attend(q[0, 0, 4 * g:4 * g + 4], k[0, 0, g], v[0, 0, g])
        check_attention(out[0, 0, 4 * g:4 * g + 4], o, f"full decode row {g}")


def test_host_buffer_step_equals_device_step():
    import torch
    from paper_2608_08878_gb300 import dc
    wl = synth.MISTRAL_1L.with_(prompt_len=1000, budget=300)
    a, b = LockStep(wl, []), LockStep(wl, [])
    a.load_prompt()
    b.load_prompt()
    for s in range(3):
        q, kn, vn = synth.step_all(wl, s)
        f = lambda x: torch.from_numpy(x.view(np.int16)).view(torch.bfloat16)
        out_h = torch.empty(q.shape, dtype=torch.float32).pin_memory()
        a.cache.decode_step_host(f(q).pin_memory(), f(kn).pin_memory(), f(vn).pin_memory(), out_h)
        out_d = b.cache.decode_step(f(q).cuda(), f(kn).cuda(), f(vn).cuda())
        assert torch.equal(out_h, out_d.cpu())
        a.cache.evict()
        b.cache.evict()
        for which in (dc.BUF_POS, dc.BUF_SCORE):
            assert torch.equal(a.cache.buffer(which), b.cache.buffer(which))


def test_errors_leave_the_cache_usable():
    import torch
    from paper_2608_08878_gb300 import dc
    cache = dc.DistillCache(1, 2, 64, 10, 4, q_heads=4)
    k = torch.zeros((1, 1, 2, 11, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(dc.DCError) as e:
        cache.append(k, k)
    assert e.value.status == dc.DC_ERR_CAPACITY
    with pytest.raises(dc.DCError) as e:
        cache.evict()
    assert e.value.status == dc.DC_ERR_STATE
    cache.append(k[:, :, :, :9].contiguous(), k[:, :, :, :9].contiguous())
    q = torch.zeros((1, 1, 4, 64), dtype=torch.bfloat16, device="cuda")
    kn = torch.zeros((1, 1, 2, 64), dtype=torch.bfloat16, device="cuda")
    cache.decode_step(q, kn, kn)
    with pytest.raises(dc.DCError) as e:
        cache.decode_step(q, kn, kn)
    assert e.value.status == dc.DC_ERR_CAPACITY
    cache.evict()
    assert cache.length() == (4, 10)
    cache.sync()


@pytest.mark.parametrize("engine", ENGINES)
def test_full_stack_sampled_rows(engine):
    """Mistral-7B 32 layers, batch 8, 32K context, budget 8192 at full size: the
    prompt-compression step and 71 steady steps, 3 sampled rows (among them the
    last row, which falls in the fused grid's split last wave). Queries leave
    the w = 64 window from step 64 on; every step from 62 on is checked, so the
    departing-query subtraction is compared with the oracle at this shape."""
    wl = synth.MISTRAL_FULL
    assert wl.window == 64
    ls = LockStep(wl, [0, 1029, wl.rows - 1], engine=engine, device_inputs=True)
    ls.load_prompt()
    for s in range(72):
        ls.step(check=(s < 3 or s % 16 == 0 or s >= 62))
    assert ls.cache.length()[0] == wl.budget


@pytest.mark.parametrize("layers,batch,kv_heads,prompt_len,budget", [
    (1, 1, 4, 8192, 2048),     # few rows: halves over two CTAs each
    (5, 8, 4, 8192, 8192),     # 160 rows: the split last wave; rows past the on-chip logits
    (2, 10, 8, 3000, 1000),    # 160 rows within the on-chip logits, many-eviction first step
])
def test_group8_rows_match_oracle(layers, batch, kv_heads, prompt_len, budget):
    """Eight query heads per KV head on the fused engine: a 32-row query tile,
    seven TMEM logit columns per tile (24 tiles on chip, then all eight
    logits through HBM), both 16-byte halves of the PV operand; the prompt
    compression and steps past a small window, sampled rows."""
    wl = synth.MISTRAL_1L.with_(layers=layers, batch=batch, kv_heads=kv_heads, q_heads=8 * kv_heads,
                                prompt_len=prompt_len, budget=budget, window=4, steps=8)
    rows = sorted({0, wl.rows // 2, wl.rows - 1})
    ls = LockStep(wl, rows, engine=2, device_inputs=True)
    assert ls.cache.engine() == "fused"
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()
    assert ls.cache.length()[0] == min(wl.prompt_len + wl.steps, wl.budget)


@pytest.mark.parametrize("batch,ctx,ratio", [(1, 4096, 0.10), (64, 4096, 0.25), (4, 16384, 0.50),
                                              (1, 32768, 0.50)])
def test_sweep_points_sampled_rows(batch, ctx, ratio):
    """Points of the throughput sweep (32 layers, Mistral-7B KV heads) at full
    size in the engine auto-selection the sweep uses: prompt compression and
    steady steps, 3 sampled rows. The first two points run on row pairs; the
    last point's budget (16384) is past the on-chip logit capacity, so its
    logits and scores go through HBM."""
    wl = synth.sweep_point(batch, ctx, ratio)
    ls = LockStep(wl, [0, wl.rows // 2 + 3, wl.rows - 1], engine=0, device_inputs=True)
    ls.load_prompt()
    for _ in range(3):
        ls.step()
    assert ls.cache.length()[0] == wl.budget


def test_aggressive_sampled_rows():
    """32 layers, batch 16, 32K context, budget 3277 (10%), hot sets reshuffled
    every 16 steps: 72 steps cross four reshuffles and the w = 64 window's
    departures; 2 sampled rows, checked around each reshuffle and at every
    step from 62 on."""
    wl = synth.AGGRESSIVE
    assert wl.epoch_len == 16 and wl.window == 64
    ls = LockStep(wl, [7, wl.rows - 3], engine=0, device_inputs=True)  # auto: fused steady steps
    ls.load_prompt()
    for s in range(72):
        ls.step(check=(s < 2 or s % 16 in (0, 1, 15) or s >= 62))
    assert ls.cache.length()[0] == wl.budget


@pytest.mark.parametrize("engine", ENGINES)
@pytest.mark.parametrize("scorer", [0, 1, 2])
def test_global_token_mode(engine, scorer):
    """Global token mode: features pooled over all heads and layers of each
    sequence, one score and one selection per sequence, every row pruned
    alike; prompt compression and steps past the window, all sequences."""
    wl = synth.MISTRAL_1L.with_(layers=3, batch=2, kv_heads=2, q_heads=8, prompt_len=400, budget=150,
                                steps=70, window=6)
    ls = SeqLockStep(wl, range(wl.batch), scorer=scorer, engine=engine)
    assert ls.cache.engine() == ("fused" if engine == 2 else "split")
    ls.load_prompt()
    for s in range(wl.steps):
        ls.step(check=(s < 3 or s % 16 == 0 or s >= 66))
    assert ls.cache.length()[0] == wl.budget


def test_global_token_mode_full_shape_sampled():
    """The same at the Mistral-7B shape (32 layers x 8 KV heads = 256 rows per
    sequence), a 2K prompt compressed to 512, then a steady step."""
    wl = synth.MISTRAL_1L.with_(layers=32, batch=1, prompt_len=2048, budget=512, steps=2)
    ls = SeqLockStep(wl, [0])
    assert ls.cache.engine() == "fused"
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()


def test_full_decode_with_split_rows_matches_oracle():
    """The full-cache comparator (the fused kernel's attention-only variant)
    with the last wave's rows split over CTA pairs: sampled rows, split and
    whole, against the oracle's plain attention."""
    import oracle
    wl, sms = _tail_workload(prompt_len=2500)
    ls = LockStep(wl, [], engine=2)
    ls.load_prompt()
    q, _, _ = ls._inputs(0)
    out = ls.cache.full_decode(q).cpu().numpy()
    qh = q.view(__import__("torch").int16).cpu().numpy().view(np.uint16)
    for r in (0, sms - 1, sms, wl.rows - 1):
        layer, b, g = wl.row_coords(r)
        k, v = synth.prompt_row(wl, layer, b, g)
        G = wl.group
        o, _ = oracle.attend(qh[layer, b, g * G:(g + 1) * G], k, v)
        check_attention(out[layer, b, g * G:(g + 1) * G], o, f"full decode row {r}")


def test_global_token_mode_with_split_rows():
    """Global token mode on the fused engine with more rows than SMs, so the
    last wave's rows are split over CTA pairs: one 160-row sequence."""
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    layers = sms // 8 + 1
    wl = synth.MISTRAL_1L.with_(layers=layers, batch=1, prompt_len=600, budget=250, steps=4, window=3)
    assert 0 < wl.rows - sms <= sms // 2
    ls = SeqLockStep(wl, [0], engine=2)
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()


def test_async_host_steps_equal_device_steps():
    """dc_step_host_async queued back to back (one sync at the end) gives the
    same outputs and cache as dc_step on device buffers."""
    import torch
    from paper_2608_08878_gb300 import dc
    wl = synth.MISTRAL_1L.with_(prompt_len=1000, budget=300)
    a, b = LockStep(wl, [], engine=2), LockStep(wl, [], engine=2)
    a.load_prompt()
    b.load_prompt()
    f = lambda x: torch.from_numpy(x.view(np.int16)).view(torch.bfloat16)
    outs, refs, keep = [], [], []
    for s in range(8):
        q, kn, vn = synth.step_all(wl, s)
        hq, hk, hv = f(q).pin_memory(), f(kn).pin_memory(), f(vn).pin_memory()
        keep.append((hq, hk, hv))
        out_h = torch.empty(q.shape, dtype=torch.float32).pin_memory()
        if s == 5:
            # the synchronous call shares the first staging set with copies
            # of the asynchronous ones still in flight
            a.cache.step_host(hq, hk, hv, out_h)
        else:
            a.cache.step_host_async(hq, hk, hv, out_h)
        outs.append(out_h)
        refs.append(b.cache.step(f(q).cuda(), f(kn).cuda(), f(vn).cuda()).cpu())
    a.cache.sync()
    for s in range(8):
        assert torch.equal(outs[s], refs[s]), s
    for which in (dc.BUF_K, dc.BUF_POS, dc.BUF_S):
        assert torch.equal(a.cache.buffer(which), b.cache.buffer(which))


def _boundary_workload(kind, budget):
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    batch = {"few": 1, "pairs": sms // 2}[kind]  # 8 rows, or 4 rows per SM
    # prompt = budget: every step appends one token and evicts one, n = budget + 1
    return synth.MISTRAL_1L.with_(batch=batch, prompt_len=budget, budget=budget, steps=3, window=4)


@pytest.mark.parametrize("kind,budget,engine", [
    ("few", 1535, "fused"),         # 12 whole tiles: every row in halves, no ragged tile
    ("few", 1536, "fused"),         # 13 tiles in halves, half 1 ends on a 1-token tile
    ("few", 127, "fused"),          # one whole tile
    ("few", 16, "fused"),           # one tile of 17 tokens: two 16-token boxes
    ("pairs", 2687, "fused-pairs"),  # 21 whole tiles, the longest row pairs take
    ("pairs", 15, "fused-pairs"),    # one tile of 16 tokens: one box
    ("pairs", 2688, "fused"),        # 22 tiles: whole rows, a 1-token ragged tile
])
def test_work_item_boundaries(kind, budget, engine):
    """The fused engine's work items at their boundaries (halves for few rows
    from 12 tiles, row pairs up to 21 tiles, a row's ragged last tile loaded in
    16-token boxes): sampled rows against the oracle over steps past the
    window, and dc_step's in-kernel eviction bit-identical to dc_decode_step
    and dc_evict."""
    import torch
    from paper_2608_08878_gb300 import dc
    wl = _boundary_workload(kind, budget)
    rows = [0, wl.rows // 2 + 1, wl.rows - 1]
    ls = LockStep(wl, rows, engine=0, device_inputs=True)
    assert ls.cache.engine(budget + 1) == engine
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()
    a, b = LockStep(wl, [], engine=0, device_inputs=True), LockStep(wl, [], engine=0, device_inputs=True)
    for x in (a, b):
        x.load_prompt()
    for s in range(wl.steps + 4):
        q, kn, vn = a._inputs(s)
        oa = a.cache.step(q, kn, vn)
        ob = b.cache.decode_step(q, kn, vn)
        b.cache.evict()
        a.cache.sync()
        b.cache.sync()
        assert torch.equal(oa, ob), s
        n = a.cache.length()[0]
        assert n == b.cache.length()[0] == budget
        for which in (dc.BUF_K, dc.BUF_V, dc.BUF_POS, dc.BUF_S, dc.BUF_Z, dc.BUF_VNORM):
            assert torch.equal(a.cache.buffer(which)[:, :n], b.cache.buffer(which)[:, :n]), (s, which)


def test_bounded_waits_give_up_and_leave_the_context_usable():
    """A wait that nothing will satisfy (a flag nothing sets, an mbarrier
    nothing arrives on) gives up after its limit, records where, and the
    kernel returns; the CUDA context and a cache built afterwards still work."""
    import torch
    from paper_2608_08878_gb300 import dc
    res = dc.wait_selftest(limit_ms=20)
    assert res["flag_gave_up"] and res["barrier_gave_up"], res
    assert res["site"] == 901, res  # the first timeout of the launch: the flag wait
    assert res["flag_wait_us"] >= 20000 and res["barrier_wait_us"] >= 20000, res
    assert res["flag_wait_us"] < 2000000 and res["barrier_wait_us"] < 2000000, res
    wl = synth.TINY.with_(steps=2)
    ls = LockStep(wl, range(wl.rows), engine=2)
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()


def _random_shapes(count=24, seed=2026, groups=(1, 2, 4)):
    """Seeded shapes over the engines' parameters (group, head size, window,
    alpha mode, engine, rows from a few to several waves, lengths from one
    token to past the row-pair limit)."""
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(count):
        group = int(rng.choice(list(groups)))
        head_dim = int(rng.choice([64, 128]))
        kv_heads = int(rng.choice([1, 2, 8]))
        layers = int(rng.integers(1, 5))
        batch = int(rng.integers(1, 640 // (layers * kv_heads) + 1))
        prompt = int(rng.integers(1, 3000))
        budget = int(rng.integers(1, prompt + 40))
        out.append(dict(group=group, head_dim=head_dim, kv_heads=kv_heads, layers=layers, batch=batch,
                        prompt_len=prompt, budget=budget, window=int(rng.choice([1, 2, 4, 8])),
                        alpha_mode=int(rng.integers(0, 2)), engine=int(rng.choice([0, 1, 2])),
                        steps=int(rng.integers(3, 7))))
    return out


@pytest.mark.parametrize("shape", _random_shapes() + _random_shapes(count=12, seed=88, groups=(8,)),
                         ids=lambda s: "L{layers}b{batch}h{kv_heads}g{group}d{head_dim}"
                         "p{prompt_len}B{budget}w{window}a{alpha_mode}e{engine}".format(**s))
def test_random_shapes_match_oracle(shape):
    """Seeded random shapes against the oracle on sampled rows: whatever
    schedule the engine picks (split, whole rows, halves, row pairs, ragged
    tiles), the step's outputs, features, scores and kept sets agree."""
    sh = dict(shape)
    engine, group = sh.pop("engine"), sh.pop("group")
    wl = synth.MISTRAL_1L.with_(q_heads=sh["kv_heads"] * group, **sh)
    rows = sorted({0, wl.rows // 2, wl.rows - 1})
    ls = LockStep(wl, rows, engine=engine, device_inputs=True, capacity=max(wl.prompt_len, wl.budget) + 16)
    ls.load_prompt()
    for _ in range(wl.steps):
        ls.step()
    assert ls.cache.length()[0] == min(wl.prompt_len + wl.steps, wl.budget)


@pytest.mark.parametrize("shape", _random_shapes(count=12, seed=7) + _random_shapes(count=6, seed=89, groups=(8,)),
                         ids=lambda s: "L{layers}b{batch}h{kv_heads}g{group}"
                         "d{head_dim}p{prompt_len}B{budget}w{window}a{alpha_mode}e{engine}".format(**s))
def test_random_shapes_step_equals_decode_then_evict(shape):
    """Seeded random shapes: dc_step (the fused engine's in-kernel select and
    compaction wherever it applies) leaves the same output and cache, bit for
    bit, as dc_decode_step followed by dc_evict."""
    import torch
    from paper_2608_08878_gb300 import dc
    sh = dict(shape)
    engine, group = sh.pop("engine"), sh.pop("group")
    wl = synth.MISTRAL_1L.with_(q_heads=sh["kv_heads"] * group, **sh)
    cap = max(wl.prompt_len, wl.budget) + 16
    a = LockStep(wl, [], engine=engine, device_inputs=True, capacity=cap)
    b = LockStep(wl, [], engine=engine, device_inputs=True, capacity=cap)
    for x in (a, b):
        x.load_prompt()
    for s in range(wl.steps):
        q, kn, vn = a._inputs(s)
        oa = a.cache.step(q, kn, vn)
        ob = b.cache.decode_step(q, kn, vn)
        b.cache.evict()
        a.cache.sync()
        b.cache.sync()
        assert torch.equal(oa, ob), s
        n = a.cache.length()[0]
        assert n == b.cache.length()[0]
        for which in (dc.BUF_K, dc.BUF_V, dc.BUF_POS, dc.BUF_S, dc.BUF_Z, dc.BUF_VNORM):
            assert torch.equal(a.cache.buffer(which)[:, :n], b.cache.buffer(which)[:, :n]), (s, which)
