"""The allocation-free attention entry point (dc_attend_noalloc), for callers
that cannot call cudaMalloc (runtimes that reserve all device memory up front,
paths that cannot take the implicit synchronisation of cudaMalloc/cudaFree).
It is called through the C ABI and checked against the handle-based
full-cache decode on the same inputs, twice in a row: the two calls share the
library's fixed scratch array, so the second one also shows that nothing left
there by the first changes its result. Kept in the last-collected file so that
a failure here does not stop the rest of the suite."""

import numpy as np
import pytest

from paper_2608_08878_gb300 import synth

import oracle
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


@pytest.mark.parametrize("head_dim", [64, 128])
@pytest.mark.parametrize("group", [1, 2, 4, 8])
@pytest.mark.parametrize("n", [1, 100, 257])
def test_noalloc_attention_matches_oracle(head_dim, group, n):
    """Every <head_dim, group> variant the entry point dispatches to, on rows of
    one token, of less than one 128-token tile and of a ragged third tile,
    against the fp64 oracle's softmax attention, twice in a row (the second
    call finds the first one's partials in the shared scratch array)."""
    import torch
    from paper_2608_08878_gb300 import dc
    rows = 3
    wl = synth.TINY.with_(kv_heads=rows, q_heads=rows * group, head_dim=head_dim, prompt_len=n,
                          seed=100 + n + group)
    k, v = synth.prompt_all(wl)                          # [1][1][rows][n][d]
    kr, vr = _bf16(torch, k).reshape(rows, n, head_dim), _bf16(torch, v).reshape(rows, n, head_dim)
    for step in (0, 1):
        q, _, _ = synth.step_all(wl, step)               # [1][1][rows * group][d]
        qh = q.reshape(rows, group, head_dim)
        out = dc.attend_noalloc(_bf16(torch, qh), kr, vr)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        for r in range(rows):
            ref, _ = oracle.attend(qh[r], k[0, 0, r], v[0, 0, r])
            check_attention(got[r], ref, f"d {head_dim} G {group} n {n} row {r} call {step}")


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

