"""The allocation-free attention entry point (dc_attend_noalloc), called
through the C ABI, against the handle-based full-cache decode on the same
inputs, twice in a row (the two calls share the library's fixed scratch
array). Kept in the last-collected file so that a failure here does not stop
the rest of the suite."""

import numpy as np
import pytest

from paper_2608_08878_gb300 import synth

from harness import check_attention

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_08878_gb300 import build
    build.build()
    import torch
    torch.cuda.init()


def _bf16(torch, a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).cuda()


def test_noalloc_attention_matches_full_decode_on_consecutive_calls():
    import torch
    from paper_2608_08878_gb300 import dc
    wl = synth.MISTRAL_1L.with_(prompt_len=1500, batch=2)
    k, v = synth.prompt_all(wl)                          # [L][b][kvh][T][d]
    kt, vt = _bf16(torch, k), _bf16(torch, v)
    rows, G, d, T = wl.rows, wl.group, wl.head_dim, wl.prompt_len
    cache = dc.DistillCache(wl.layers, wl.kv_heads, d, T + 1, 100, batch=wl.batch)
    cache.append(kt, vt)
    kr, vr = kt.reshape(rows, T, d), vt.reshape(rows, T, d)
    for step in (0, 1):
        q, _, _ = synth.step_all(wl, step)               # [L][b][qh][d]
        qt = _bf16(torch, q)
        ref = cache.full_decode(qt)
        out = dc.attend_noalloc(qt.reshape(rows, G, d), kr, vr)
        torch.cuda.synchronize()
        check_attention(out.reshape(ref.shape).cpu().numpy(), ref.cpu().numpy(), f"call {step}")


def test_noalloc_rejects_oversized_and_bad_shapes():
    import torch
    from paper_2608_08878_gb300 import dc
    q = torch.zeros((40000, 8, 128), dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros((40000, 1, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(dc.DCError) as e:   # 40000 * 8 * 132 * 4 bytes > 16 MiB
        dc.attend_noalloc(q, kv, kv)
    assert e.value.status == dc.DC_ERR_CAPACITY and "scratch" in str(e.value)
    with pytest.raises(dc.DCError) as e:
        dc.attend_noalloc(q[:4, :3], kv[:4], kv[:4])  # group 3
    assert e.value.status == dc.DC_ERR_INVALID_ARG


def test_noalloc_attention_replays_in_a_cuda_graph():
    """dc_attend_noalloc keeps no state between calls, so a stream capture of
    it replays as the same computation on whatever the captured buffers hold:
    replays with new queries equal eager calls bit for bit."""
    import torch
    from paper_2608_08878_gb300 import dc
    wl = synth.MISTRAL_1L.with_(prompt_len=700)
    k, v = synth.prompt_all(wl)
    rows, G, d, T = wl.rows, wl.group, wl.head_dim, wl.prompt_len
    kr, vr = _bf16(torch, k).reshape(rows, T, d), _bf16(torch, v).reshape(rows, T, d)
    q_static = _bf16(torch, synth.step_all(wl, 0)[0]).reshape(rows, G, d).clone()
    out_static = torch.empty((rows, G, d), dtype=torch.float32, device="cuda")
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):  # warm-up outside the capture
        dc.attend_noalloc(q_static, kr, vr, out=out_static)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        dc.attend_noalloc(q_static, kr, vr, out=out_static)
    for step in (1, 2, 3):
        q = _bf16(torch, synth.step_all(wl, step)[0]).reshape(rows, G, d)
        q_static.copy_(q)
        graph.replay()
        ref = dc.attend_noalloc(q, kr, vr)
        torch.cuda.synchronize()
        assert torch.equal(out_static, ref), step
