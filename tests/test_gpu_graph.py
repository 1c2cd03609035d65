"""Graph mode (device-counted steps): dc_step with its step arguments advanced
on the device equals ordinary dc_step calls bit for bit, eagerly and when one
captured step is replayed from a CUDA graph as the following steps."""

import numpy as np
import pytest

from paper_2608_08878_gb300 import synth

pytestmark = pytest.mark.gpu

BUFS = ("BUF_K", "BUF_V", "BUF_POS", "BUF_S", "BUF_Z", "BUF_VNORM")


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_08878_gb300 import build
    build.build()
    import torch
    torch.cuda.init()


def _pair(wl, stream=None):
    """Two caches of the same workload with the prompt loaded."""
    from paper_2608_08878_gb300 import dc, synth_device
    out = []
    for _ in range(2):
        c = dc.DistillCache(wl.layers, wl.kv_heads, wl.head_dim, wl.prompt_len + 8, wl.budget, batch=wl.batch,
                            q_heads=wl.q_heads, window=wl.window, mlp_hidden=wl.mlp_hidden, layernorm=wl.layernorm,
                            engine=2, seed=wl.policy_seed, stream=stream)
        k, v = synth_device.prompt(wl, 0, wl.prompt_len)
        c.append(k, v)
        out.append(c)
    return out


def _same_cache(a, b):
    import torch
    from paper_2608_08878_gb300 import dc
    n = a.length()[0]
    assert a.length() == b.length()
    for name in BUFS:
        which = getattr(dc, name)
        assert torch.equal(a.buffer(which)[:, :n], b.buffer(which)[:, :n]), name


def _rows_for_sms(per_sm_times, extra):
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    return (per_sm_times * sms + extra) // 8


@pytest.mark.parametrize("case", ["few rows", "few rows in halves", "last wave in halves", "long rows", "row pairs"])
def test_graph_mode_steps_equal_ordinary_steps(case):
    import torch
    from paper_2608_08878_gb300 import synth_device
    batch, prompt = {"few rows": (1, 600), "few rows in halves": (1, 2000),
                     "last wave in halves": (_rows_for_sms(1, 8), 600), "long rows": (1, 9000),
                     "row pairs": (_rows_for_sms(4, 0), 600)}[case]
    wl = synth.MISTRAL_1L.with_(batch=batch, prompt_len=prompt, budget=prompt, window=4)
    a, b = _pair(wl)
    if case == "row pairs":
        assert a.engine(prompt + 1) == "fused-pairs"
    s = 0
    for _ in range(wl.window + 1):  # a full window of decode steps first
        q, kn, vn = synth_device.step_inputs(wl, s)
        a.step(q, kn, vn)
        b.step(q, kn, vn)
        s += 1
    b.set_graph_mode(True)
    for _ in range(2 * wl.window + 3):  # past the window: the counted slots wrap
        q, kn, vn = synth_device.step_inputs(wl, s)
        oa = a.step(q, kn, vn)
        ob = b.step(q, kn, vn)
        torch.cuda.synchronize()
        assert torch.equal(oa, ob), s
        s += 1
    b.set_graph_mode(False)
    a.sync()
    b.sync()
    _same_cache(a, b)
    for _ in range(3):  # ordinary steps again from the state the device counted
        q, kn, vn = synth_device.step_inputs(wl, s)
        assert torch.equal(a.step(q, kn, vn), b.step(q, kn, vn)), s
        s += 1
    a.sync()
    b.sync()
    _same_cache(a, b)


@pytest.mark.parametrize("rows_per_sm,prompt", [(0, 700), (0, 2000), (4, 700)])  # whole rows; halves
def test_graph_mode_replays_a_captured_step_as_the_next_steps(rows_per_sm, prompt):  # (cooperative); pairs
    import torch
    from paper_2608_08878_gb300 import synth_device
    batch = _rows_for_sms(rows_per_sm, 0) if rows_per_sm else 1
    wl = synth.MISTRAL_1L.with_(batch=batch, prompt_len=prompt, budget=prompt, window=4)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        a, b = _pair(wl, stream=stream)
        s = 0
        for _ in range(wl.window + 1):
            q, kn, vn = synth_device.step_inputs(wl, s)
            a.step(q, kn, vn)
            b.step(q, kn, vn)
            s += 1
        b.set_graph_mode(True)
        q, kn, vn = synth_device.step_inputs(wl, s)  # one eager step first (kernel attributes set)
        assert torch.equal(a.step(q, kn, vn), b.step(q, kn, vn))
        s += 1
        q0, k0, v0 = synth_device.step_inputs(wl, s)
        sq, sk, sv = q0.clone(), k0.clone(), v0.clone()
        out = torch.empty(q0.shape, dtype=torch.float32, device="cuda")
        graph = torch.cuda.CUDAGraph()
        stream.synchronize()
        with torch.cuda.graph(graph, stream=stream):
            b.step(sq, sk, sv, out=out)  # captured, not run
        for _ in range(2 * wl.window + 3):
            q, kn, vn = synth_device.step_inputs(wl, s)
            sq.copy_(q)
            sk.copy_(kn)
            sv.copy_(vn)
            graph.replay()
            ref = a.step(q, kn, vn)
            stream.synchronize()
            assert torch.equal(out, ref), s
            s += 1
        b.set_graph_mode(False)
        a.sync()
        b.sync()
        _same_cache(a, b)


def test_graph_mode_guards():
    from paper_2608_08878_gb300 import dc, synth_device
    wl = synth.MISTRAL_1L.with_(prompt_len=300, budget=300, window=4)
    a, _ = _pair(wl)
    with pytest.raises(dc.DCError) as e:  # no window of decode steps yet
        a.set_graph_mode(True)
    assert e.value.status == dc.DC_ERR_STATE
    for s in range(wl.window):
        a.step(*synth_device.step_inputs(wl, s))
    a.set_graph_mode(True)
    q, kn, vn = synth_device.step_inputs(wl, 99)
    for call in (lambda: a.decode_step(q, kn, vn), lambda: a.evict(), lambda: a.append(kn[..., None, :], vn[..., None, :]),
                 lambda: a.full_decode(q)):
        with pytest.raises(dc.DCError) as e:
            call()
        assert e.value.status == dc.DC_ERR_STATE
    with pytest.raises(dc.DCError) as e:
        a.step(q, kn, vn, budget=7)
    assert e.value.status == dc.DC_ERR_INVALID_ARG
    a.set_graph_mode(False)
    a.step(q, kn, vn)
    a.sync()
