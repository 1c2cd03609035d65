"""Failure paths and debug-build checks that need no GPU fault.

* Allocation failures: a create that cannot fit in HBM, and a failure injected
  at each device allocation of a create (a host-side hook, no real shortage),
  return DC_ERR_OOM after freeing what they took; the next create works. A
  later call that needs a new buffer fails with DC_ERR_OOM and leaves the
  handle usable.
* The debug build (device-side index checks, guard regions around every
  buffer of a handle, both checked by dc_sync): its self-tests, and the small
  parity cases run against it in a child process (any failed index check or
  damaged guard makes dc_sync raise there).
"""

import os
import subprocess
import sys

import numpy as np
import pytest

from paper_2608_08878_gb300 import synth

from harness import LockStep

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_08878_gb300 import build
    build.build()
    import torch
    torch.cuda.init()


def _free_bytes():
    import torch
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info()[0]


def test_create_too_large_for_hbm_is_oom_and_frees_what_it_took():
    from paper_2608_08878_gb300 import dc
    before = _free_bytes()
    # 16384 rows x 40064 slots x 128 dims: K and V 168 GB each, more than the GPU holds
    with pytest.raises(dc.DCError) as e:
        dc.DistillCache(32, 8, 128, 40000, 8192, batch=64)
    assert e.value.status == dc.DC_ERR_OOM, str(e.value)
    assert abs(_free_bytes() - before) < (64 << 20)
    wl = synth.TINY
    ls = LockStep(wl, range(wl.rows), engine=2)
    ls.load_prompt()
    for _ in range(3):
        ls.step()


def test_injected_allocation_failure_at_every_allocation_of_a_create():
    """The hook fails the nth allocation of the next create, for every n until
    a create gets through: each failed create returns DC_ERR_OOM, the device
    memory it took comes back, and the create after it works."""
    from paper_2608_08878_gb300 import dc
    wl = synth.MISTRAL_1L.with_(prompt_len=300, budget=100)
    before = _free_bytes()
    failures = 0
    for nth in range(64):
        dc.debug_fail_alloc(nth)
        try:
            c = dc.DistillCache(wl.layers, wl.kv_heads, wl.head_dim, 400, wl.budget, q_heads=wl.q_heads,
                                engine=2)
        except dc.DCError as e:
            assert e.status == dc.DC_ERR_OOM, (nth, str(e))
            assert abs(_free_bytes() - before) < (64 << 20), nth
            failures += 1
            continue
        dc.debug_fail_alloc(-1)
        assert c.engine(301) == "fused"
        c.close()
        break
    else:
        pytest.fail("no create got through")
    assert failures >= 20  # every buffer of the handle was a failure point
    dc.debug_fail_alloc(-1)
    ls = LockStep(wl, [0, 5], engine=2)
    ls.load_prompt()
    for _ in range(3):
        ls.step()


def test_allocation_failure_after_creation_leaves_the_handle_usable():
    """Per-row budgets and the asynchronous host path allocate on first use:
    a failure there is DC_ERR_OOM, nothing changes, and the same call works
    once memory is available again."""
    import torch
    from paper_2608_08878_gb300 import dc
    wl = synth.TINY.with_(steps=6)
    ls = LockStep(wl, range(wl.rows), engine=2)
    ls.load_prompt()
    ls.step()
    dc.debug_fail_alloc(1)
    with pytest.raises(dc.DCError) as e:
        ls.cache.set_row_budgets(np.full(wl.rows, wl.budget, dtype=np.int32))
    assert e.value.status == dc.DC_ERR_OOM
    ls.step()  # the handle still steps, in lock step with the oracle
    q, kn, vn = ls._inputs(ls.step_idx)
    host = [x.cpu().pin_memory() for x in (q, kn, vn)]
    out = torch.empty(q.shape, dtype=torch.float32).pin_memory()
    dc.debug_fail_alloc(0)
    with pytest.raises(dc.DCError) as e:
        ls.cache.step_host_async(*host, out)
    assert e.value.status == dc.DC_ERR_OOM
    assert ls.cache.length()[1] == wl.prompt_len + 2  # the step did not happen
    ls.cache.set_row_budgets(np.full(wl.rows, wl.budget, dtype=np.int32))
    ls.cache.set_row_budgets(None)
    ls.cache.step_host_async(*host, out)
    ls.cache.sync()
    dc.debug_fail_alloc(-1)


def test_debug_build_checks_and_small_parity_cases():
    """Builds the debug library, then in a child process with DC_LIBRARY=debug:
    the index-check self-test, a damaged guard region reported by dc_sync,
    and the small parity cases (every dc_sync there checks the index-check
    status and every guard region)."""
    from paper_2608_08878_gb300 import build
    build.build_debug()
    env = dict(os.environ, DC_LIBRARY="debug")
    cases = ("not full_stack and not aggressive and not sweep_points and not full_shape and not "
             "mistral_single_layer and not device_generator")
    cmd = [sys.executable, "-m", "pytest", "-x", "-q", "-m", "gpu",
           os.path.join(ROOT, "tests", "debug_build_checks.py"),
           os.path.join(ROOT, "tests", "test_gpu_parity.py"), "-k", cases]
    res = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    assert res.returncode == 0, res.stdout[-4000:] + res.stderr[-2000:]
    assert " passed" in res.stdout
