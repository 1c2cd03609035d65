"""Host-side checks of the C ABI library (no GPU): it loads, exports every
function the header declares, validates arguments before touching the device,
and its seeded policy initialisation matches the input generator bit for bit."""

import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2608_08878_gb300 import dc, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_08878_gb300 import build
    build.build()


def header_functions():
    names = set()
    inc = os.path.join(ROOT, "include")
    for f in os.listdir(inc):
        if f.endswith(".h"):
            text = open(os.path.join(inc, f)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(dc_[a-z_0-9]+)\s*\(", text))
    return names


def test_library_exports_every_declared_function():
    L = dc.lib()
    declared = header_functions()
    assert declared, "no declarations found"
    for name in sorted(declared):
        assert hasattr(L, name), f"{name} is declared but not exported"
    assert declared <= set(dc.EXPORTS) | set(), sorted(declared - set(dc.EXPORTS))


def test_policy_init_matches_generator():
    for seed, H in [(0, 128), (0, 64), (7, 32), (123456789, 256), (1, 5)]:
        np.testing.assert_array_equal(dc.policy_init(seed, H), synth.policy_weights(seed, H))
    assert dc.policy_blob_len(128) == 9 * 128 + 1


def test_config_defaults():
    cfg = dc.dc_config()
    assert dc.lib().dc_config_default(C.byref(cfg)) == dc.DC_OK
    assert (cfg.batch, cfg.q_heads, cfg.window, cfg.mlp_hidden, cfg.layernorm, cfg.alpha_mode,
            cfg.engine, cfg.keep_features, cfg.seed) == (1, 0, 64, 128, 1, 0, 0, 0, 0)
    assert (cfg.tail_split, cfg.scorer, cfg.n_sinks, cfg.budget_ratio, cfg.budget_min,
            cfg.budget_basis) == (1, 0, 4, 0.0, 32, 0)
    assert dc.lib().dc_config_default(None) == dc.DC_ERR_INVALID_ARG


@pytest.mark.parametrize("args,field", [
    ((1, 8, 96, 100, 10), "head_dim"),
    ((1, 8, 128, 10, 10), "budget"),
    ((1, 8, 128, 10, 0), "budget"),
    ((0, 8, 128, 100, 10), "layers"),
])
def test_create_rejects_bad_shapes_without_touching_the_device(args, field):
    h = C.c_void_p()
    st = dc.lib().dc_cache_create(*args, None, C.byref(h))
    assert st == dc.DC_ERR_INVALID_ARG and not h.value
    assert field in dc.lib().dc_last_error(None).decode()


def test_create_rejects_bad_config():
    L = dc.lib()
    for field, value in [("q_heads", 12), ("window", 0), ("mlp_hidden", 100), ("alpha_mode", 2),
                         ("engine", 5), ("scorer", 3), ("n_sinks", -1), ("budget_ratio", 1.5),
                         ("budget_min", 0), ("budget_basis", 2)]:
        cfg = dc.dc_config()
        L.dc_config_default(C.byref(cfg))
        setattr(cfg, field, value)
        h = C.c_void_p()
        assert L.dc_cache_create(1, 8, 128, 100, 10, C.byref(cfg), C.byref(h)) == dc.DC_ERR_INVALID_ARG


def test_null_handles_are_rejected():
    L = dc.lib()
    assert L.dc_cache_destroy(None) == dc.DC_OK
    assert L.dc_evict(None, 1) == dc.DC_ERR_INVALID_ARG
    assert L.dc_append(None, None, None, 0) == dc.DC_ERR_INVALID_ARG
    assert L.dc_sync(None) == dc.DC_ERR_INVALID_ARG
    assert L.dc_policy_init(0, 0, None, 0) == dc.DC_ERR_INVALID_ARG
    assert L.dc_set_graph_mode(None, 1) == dc.DC_ERR_INVALID_ARG
    assert L.dc_step_host_async(None, None, None, None, None, 0) == dc.DC_ERR_INVALID_ARG
    assert L.dc_set_row_budgets(None, None, 0) == dc.DC_ERR_INVALID_ARG
    assert L.dc_wait_selftest(1000000, None, None) == dc.DC_ERR_INVALID_ARG
    assert L.dc_wait_selftest(10, None, None) == dc.DC_ERR_INVALID_ARG


def test_training_kernels_validate_before_touching_the_device():
    L = dc.lib()
    for args in [(1, 10, 11, 1.0), (0, 10, 5, 1.0), (1, 10, 5, 0.0), (1, 10, 0, 1.0)]:
        rows, n, B, tau = args
        assert L.dc_pl_log_partition(C.c_void_p(16), rows, n, B, tau, C.c_void_p(16), None) == dc.DC_ERR_INVALID_ARG
        assert L.dc_gumbel_top_b(C.c_void_p(16), C.c_void_p(16), rows, n, B, tau, C.c_void_p(16), None, None,
                                 None) == dc.DC_ERR_INVALID_ARG
    assert L.dc_pl_log_partition(None, 1, 10, 5, 1.0, C.c_void_p(16), None) == dc.DC_ERR_INVALID_ARG
    assert b"B <= L" in L.dc_train_last_error() or b"NULL" in L.dc_train_last_error()


def test_header_compiles_as_c_and_matches_the_binding(tmp_path):
    """A C11 program includes the header, links the library and calls its
    host-only entry points; the header's dc_config layout (size and every
    field's offset) is the binding's."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    fields = [f for f, _ in dc.dc_config._fields_]
    src = tmp_path / "abi.c"
    src.write_text(
        "#include <stddef.h>\n#include <stdio.h>\n#include \"distillcache.h\"\n"
        "int main(void) {\n"
        "  dc_config cfg;\n"
        "  if (dc_config_default(&cfg) != DC_OK) return 1;\n"
        "  dc_cache* h = 0;\n"
        "  if (dc_cache_create(1, 8, 96, 100, 10, &cfg, &h) != DC_ERR_INVALID_ARG || h) return 2;\n"
        "  printf(\"%zu %zu %d %d\\n\", sizeof(dc_config), dc_policy_blob_len(128), cfg.window, cfg.mlp_hidden);\n"
        + "".join(f"  printf(\"%zu\\n\", offsetof(dc_config, {f}));\n" for f in fields)
        + "  return 0;\n}\n")
    exe = tmp_path / "abi"
    lib_dir = os.path.dirname(dc.LIB_PATH)
    subprocess.run([cc, "-std=c11", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"), str(src),
                    "-o", str(exe), "-L", lib_dir, "-ldistillcache", "-Wl,-rpath," + lib_dir], check=True,
                   capture_output=True, text=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()
    size, blob, window, hidden = (int(x) for x in out[:4])
    assert (size, blob, window, hidden) == (C.sizeof(dc.dc_config), 9 * 128 + 1, 64, 128)
    assert [int(x) for x in out[4:]] == [getattr(dc.dc_config, f).offset for f in fields]


def _unopened_cache(layers=2, batch=1, kv_heads=2, q_heads=4, head_dim=64):
    """A DistillCache object with the shape bookkeeping of a real one but no
    library handle: the binding's argument checks run before any library call,
    so they can be exercised without a GPU."""
    c = object.__new__(dc.DistillCache)
    c._h = None
    c.layers, c.batch, c.kv_heads, c.q_heads, c.head_dim = layers, batch, kv_heads, q_heads, head_dim
    c.group, c.rows, c.device = q_heads // kv_heads, layers * batch * kv_heads, 0
    return c


def test_binding_rejects_tensors_that_do_not_match_the_abi():
    """Tensors passed by pointer are checked for device or host memory, element
    type, dense layout and element count, with DC_ERR_INVALID_ARG, before the
    library is called (a wrong one would be read or written out of bounds)."""
    import torch
    c = _unopened_cache()
    q = torch.zeros((2, 1, 4, 64), dtype=torch.bfloat16)
    kn = torch.zeros((2, 1, 2, 64), dtype=torch.bfloat16)
    out = torch.zeros((2, 1, 4, 64), dtype=torch.float32)
    bad = {
        "host tensors for a device call": lambda: c.step(q, kn, kn, out),
        "host tensors for full-cache attention": lambda: c.full_decode(q, out),
        "host tensors for append": lambda: c.append(kn[..., None, :], kn[..., None, :]),
        "q of the wrong type": lambda: c.step_host(q.float(), kn, kn, out),
        "out of the wrong type": lambda: c.step_host(q, kn, kn, out.bfloat16()),
        "k_new one head short": lambda: c.step_host(q, kn[:, :, :1], kn, out),
        "q with a group too few": lambda: c.decode_step_host(q[:, :, :2].contiguous(), kn, kn, out),
        "non-contiguous out": lambda: c.step_host_async(q, kn, kn, out.transpose(2, 3)),
        "not a tensor": lambda: c.step_host(q.float().numpy(), kn, kn, out),
        "k and v of different shapes": lambda: c.append(kn[..., None, :], kn[:1, ..., None, :]),
        "attention q not 3-D": lambda: dc.attend_noalloc(q, kn, kn),
        "attention on host tensors": lambda: dc.attend_noalloc(q[0, 0, :, None], kn[0, 0, :, None], kn[0, 0, :, None]),
        "attention k of another head size": lambda: dc.attend_noalloc(
            torch.zeros((2, 2, 64), dtype=torch.bfloat16), torch.zeros((2, 5, 128), dtype=torch.bfloat16),
            torch.zeros((2, 5, 128), dtype=torch.bfloat16)),
        "attention v of another shape than k (same element count)": lambda: dc.attend_noalloc(
            torch.zeros((2, 2, 64), dtype=torch.bfloat16), torch.zeros((2, 5, 64), dtype=torch.bfloat16),
            torch.zeros((5, 2, 64), dtype=torch.bfloat16)),
        "log Z scores on the host": lambda: dc.pl_log_partition(torch.zeros((2, 10)), 3),
        "log Z scores not 2-D": lambda: dc.pl_log_partition(torch.zeros(10), 3),
        "Gumbel-top-B on the host": lambda: dc.gumbel_top_b(torch.zeros((2, 10)), torch.zeros((2, 10)), 3),
    }
    for what, call in bad.items():
        with pytest.raises(dc.DCError) as e:
            call()
        assert e.value.status == dc.DC_ERR_INVALID_ARG, what


def test_binding_accepts_host_tensors_of_the_abi_shapes(monkeypatch):
    """The host-buffer calls take CPU tensors of exactly the declared sizes in
    any shape; a well-formed call reaches the library with the tensors' own
    addresses (a stand-in library records the call)."""
    import torch
    calls = []

    class FakeLib:
        def __getattr__(self, name):
            return lambda *a: calls.append((name, a)) or dc.DC_OK

    monkeypatch.setattr(dc, "lib", lambda: FakeLib())
    c = _unopened_cache()
    q = torch.zeros((2, 1, 4, 64), dtype=torch.bfloat16)
    kn = torch.zeros((2, 1, 2, 64), dtype=torch.bfloat16)
    out = torch.zeros((2, 1, 4, 64), dtype=torch.float32)
    c.step_host(q, kn, kn, out, budget=3)
    c.decode_step_host(q.view(8, 64), kn, kn, out)
    c.step_host_async(q, kn.view(4, 64), kn, out)
    ptrs = (q.data_ptr(), kn.data_ptr(), kn.data_ptr(), out.data_ptr())
    assert calls == [("dc_step_host", (None,) + ptrs + (3,)), ("dc_decode_step_host", (None,) + ptrs),
                     ("dc_step_host_async", (None,) + ptrs + (0,))]
