"""Checks that only make sense against the debug build of the library (run by
tests/test_gpu_debug.py in a child process with DC_LIBRARY=debug; named so
that pytest does not collect it on its own)."""

import pytest

from paper_2608_08878_gb300 import synth

from harness import LockStep

pytestmark = pytest.mark.gpu


def test_the_debug_library_is_loaded():
    from paper_2608_08878_gb300 import dc
    assert dc.LIB_PATH.endswith("libdistillcache_debug.so")
    assert dc.debug_checks()


def test_index_check_fails_records_and_skips():
    from paper_2608_08878_gb300 import dc
    r = dc.debug_bounds_selftest()
    assert r == {"status": 4, "site": 903, "index": 64, "limit": 64, "skipped": True}


def test_damaged_guard_region_is_reported_by_sync():
    from paper_2608_08878_gb300 import dc
    wl = synth.TINY.with_(steps=2)
    ls = LockStep(wl, range(wl.rows), engine=2)
    ls.load_prompt()
    ls.step()
    ls.cache.sync()
    ls.cache.debug_corrupt_guard()
    with pytest.raises(dc.DCError) as e:
        ls.cache.sync()
    assert e.value.status == dc.DC_ERR_DEVICE and "guard region" in str(e.value)
