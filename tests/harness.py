"""Lock-step runner: the CUDA path (through the C ABI) and the fp64 oracle on
the same seeded inputs, compared step by step on a sample of rows."""

from __future__ import annotations

import math

import numpy as np

import oracle
from paper_2608_08878_gb300 import synth

# Tolerances (bf16 inputs, fp32 accumulation on the GPU, fp64 oracle).
ATTN_MAX_ABS = 2e-2
ATTN_REL_L2 = 1e-2
FEAT_RTOL = 1e-3
FEAT_FLOOR = 1e-3  # absolute floor as a fraction of the column's RMS over the row


def close_rel(gpu, ref, rtol, floor_frac, what):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    if ref.size == 0:
        return
    floor = floor_frac * math.sqrt(float(np.mean(ref ** 2)))
    err = np.abs(gpu - ref)
    tol = rtol * np.abs(ref) + floor
    bad = ~(err <= tol)
    if bad.any():
        i = int(np.argmax(np.where(bad, err / np.maximum(tol, 1e-300), 0)))
        raise AssertionError(f"{what}: {int(bad.sum())}/{bad.size} outside rtol {rtol} + floor {floor:.3g};"
                             f" worst at {i}: gpu {gpu.flat[i]!r} ref {ref.flat[i]!r}")


def check_attention(gpu_o, ref_o, what):
    gpu_o = np.asarray(gpu_o, dtype=np.float64)
    ref_o = np.asarray(ref_o, dtype=np.float64)
    assert gpu_o.shape == ref_o.shape, (what, gpu_o.shape, ref_o.shape)
    max_abs = float(np.max(np.abs(gpu_o - ref_o))) if ref_o.size else 0.0
    rel = float(np.linalg.norm(gpu_o - ref_o) / max(np.linalg.norm(ref_o), 1e-30))
    assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, f"{what}: max-abs {max_abs:.3g} rel-L2 {rel:.3g}"
    return max_abs, rel


class LockStep:
    """Drives a DistillCache and oracle rows for a sample of its rows."""

    def __init__(self, wl: synth.Workload, rows, *, engine=0, device_inputs=False, capacity=None,
                 tail_split=True, scorer=0, n_sinks=4, budget_ratio=0.0, budget_min=32, budget_basis=0,
                 row_budgets=None):
        import torch
        from paper_2608_08878_gb300 import dc, synth_device
        self.torch, self.dc, self.sd = torch, dc, synth_device
        self.wl = wl
        self.rows = list(rows)
        self.device_inputs = device_inputs
        cap = capacity or wl.capacity
        self.blob = synth.policy_weights(wl.policy_seed, wl.mlp_hidden)
        self.cache = dc.DistillCache(wl.layers, wl.kv_heads, wl.head_dim, cap, wl.budget,
                                     batch=wl.batch, q_heads=wl.q_heads, window=wl.window,
                                     mlp_hidden=wl.mlp_hidden, layernorm=wl.layernorm,
                                     alpha_mode=wl.alpha_mode, engine=engine, keep_features=True,
                                     seed=wl.policy_seed, tail_split=tail_split, scorer=scorer,
                                     n_sinks=n_sinks, budget_ratio=budget_ratio, budget_min=budget_min,
                                     budget_basis=budget_basis)
        self.scorer, self.n_sinks = scorer, n_sinks
        self.budget_ratio, self.budget_min, self.budget_basis = budget_ratio, budget_min, budget_basis
        self.capacity = cap
        self.cache.set_policy(self.blob)
        self.row_budgets = None if row_budgets is None else np.asarray(row_budgets, dtype=np.int32)
        if self.row_budgets is not None:
            self.cache.set_row_budgets(self.row_budgets)
        self.orows = {}
        alpha_mode = 1 if scorer == 1 else wl.alpha_mode  # H2O ranks by the cumulative mass
        for r in self.rows:
            self.orows[r] = oracle.OracleRow(wl.head_dim, wl.group, wl.window, alpha_mode, cap)
        self.step_idx = 0
        self.stats = {"attn_max_abs": 0.0, "attn_rel": 0.0, "steps": 0, "evicted": 0}

    def load_prompt(self, chunk=8192):
        wl, torch = self.wl, self.torch
        if self.device_inputs:
            for t0 in range(0, wl.prompt_len, chunk):
                T = min(chunk, wl.prompt_len - t0)
                k, v = self.sd.prompt(wl, t0, T)
                self.cache.append(k, v)
                del k, v
        else:
            k, v = synth.prompt_all(wl)
            kt = torch.from_numpy(k.view(np.int16)).view(torch.bfloat16).cuda()
            vt = torch.from_numpy(v.view(np.int16)).view(torch.bfloat16).cuda()
            self.cache.append(kt, vt)
        for r, orow in self.orows.items():
            layer, b, g = wl.row_coords(r)
            k, v = synth.prompt_row(wl, layer, b, g)
            orow.append(k, v)

    def _inputs(self, step):
        wl, torch = self.wl, self.torch
        if self.device_inputs:
            return self.sd.step_inputs(wl, step)
        q, kn, vn = synth.step_all(wl, step)
        f = lambda a: torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).cuda()
        return f(q), f(kn), f(vn)

    def _row_slice(self, which, r, n):
        return self.cache.buffer(which, r, 1)[0, :n].cpu().numpy()

    def step(self, evict=True, budget=0, check=True):
        wl, dc = self.wl, self.dc
        s = self.step_idx
        q, kn, vn = self._inputs(s)
        out = self.cache.decode_step(q, kn, vn)
        self.cache.sync()  # raises on any device-side status (e.g. a wait that gave up)
        lens = self.cache.row_lengths()
        out_h = out.cpu().numpy()
        G = wl.group
        for r, orow in self.orows.items():
            layer, b, g = wl.row_coords(r)
            qb, knb, vnb = synth.step_row(wl, s, layer, b, g)
            res = orow.step(qb, knb, vnb, self.blob, wl.mlp_hidden, wl.layernorm)
            if not check:
                continue
            n = int(lens[r])
            o_gpu = out_h[layer, b, g * G:(g + 1) * G]
            ma, rel = check_attention(o_gpu, res["o"], f"step {s} row {r} attention")
            self.stats["attn_max_abs"] = max(self.stats["attn_max_abs"], ma)
            self.stats["attn_rel"] = max(self.stats["attn_rel"], rel)
            hq = self.cache.buffer(dc.BUF_HQ, r, 1)[0].cpu().numpy()
            close_rel(hq, res["Hq"], FEAT_RTOL, 0.0, f"step {s} row {r} entropy")
            pos = self._row_slice(dc.BUF_POS, r, n)
            order = np.argsort(pos, kind="stable")
            assert np.array_equal(pos[order], res["pos"]), f"step {s} row {r}: positions differ"
            feat = self._row_slice(dc.BUF_FEAT, r, n)[order]
            names = ["alpha", "|v|", "sigma", "H", "pos"]
            for c in range(5):
                close_rel(feat[:, c], res["feat"][:, c], FEAT_RTOL, FEAT_FLOOR, f"step {s} row {r} {names[c]}")
            score = self._row_slice(dc.BUF_SCORE, r, n)[order]
            if self.scorer == 2:  # sinks, then positions relative to the newest: exact in fp32
                ref = orow.heuristic_scores(2, self.n_sinks).astype(np.float32)
                assert np.array_equal(score.astype(np.float32), ref), f"step {s} row {r} score"
            else:
                ref = res["score"] if self.scorer == 0 else orow.heuristic_scores(1)
                close_rel(score, ref, FEAT_RTOL, FEAT_FLOOR, f"step {s} row {r} score")
        if evict:
            self.evict(budget)
        self.step_idx += 1
        self.stats["steps"] += 1
        return out

    def evict(self, budget=0):
        dc = self.dc
        lens = self.cache.row_lengths()
        n, _ = self.cache.length()
        gpu_scores = {}
        for r in self.orows:
            pos = self._row_slice(dc.BUF_POS, r, int(lens[r]))
            sc = self._row_slice(dc.BUF_SCORE, r, int(lens[r]))
            order = np.argsort(pos, kind="stable")
            gpu_scores[r] = sc[order]
        self.cache.evict(budget)
        self.cache.sync()
        lens2 = self.cache.row_lengths()
        self.stats["evicted"] += int(max((lens[r] - lens2[r] for r in self.orows), default=0))
        for r, orow in self.orows.items():
            if budget > 0:
                B = budget
            elif self.row_budgets is not None:
                B = int(self.row_budgets[r])
            else:
                B = self.budget_now(n)
            assert lens2[r] == min(lens[r], B), (r, lens2[r], lens[r], B)
            orow.evict(B, gpu_scores[r])
            self.check_row_state(r, int(lens2[r]))

    def budget_now(self, n_cached):
        """The budget of the step that just ran (fixed, or the dynamic one)."""
        if self.budget_ratio <= 0:
            return self.wl.budget
        _, seen = self.cache.length()
        L = seen if self.budget_basis == 0 else n_cached
        B = max(int(math.floor(float(np.float32(self.budget_ratio)) * L)), self.budget_min)
        return min(B, self.capacity - 1)

    def check_row_state(self, r, n):
        dc = self.dc
        orow = self.orows[r]
        pos = self._row_slice(dc.BUF_POS, r, n)
        order = np.argsort(pos, kind="stable")
        assert np.array_equal(pos[order], orow.positions()), f"row {r}: retained positions differ"
        K = self.cache.buffer(dc.BUF_K, r, 1)[0, :n].view(self.torch.int16).cpu().numpy().view(np.uint16)
        V = self.cache.buffer(dc.BUF_V, r, 1)[0, :n].view(self.torch.int16).cpu().numpy().view(np.uint16)
        ok, ov = orow.kv_bits()
        assert np.array_equal(K[order], ok) and np.array_equal(V[order], ov), f"row {r}: K/V bytes differ"
        # the stored sums cover the window's queries before the last step
        S = self._row_slice(dc.BUF_S, r, n)[order]
        Z = self._row_slice(dc.BUF_Z, r, n)[order]
        oS, oZ = orow.window_sums_prior()
        close_rel(Z, oZ, FEAT_RTOL, FEAT_FLOOR, f"row {r} window mass Z")
        close_rel(S, oS, FEAT_RTOL, FEAT_FLOOR, f"row {r} window sum S")


class SeqLockStep:
    """Global token mode: drives a DistillCache with global_tokens and one
    sequence oracle per sampled sequence (rows = layers x KV heads)."""

    def __init__(self, wl: synth.Workload, seqs, *, capacity=None, scorer=0, engine=0):
        import torch
        from paper_2608_08878_gb300 import dc
        self.torch, self.dc, self.wl = torch, dc, wl
        self.seqs = list(seqs)
        cap = capacity or wl.capacity
        self.blob = synth.policy_weights(wl.policy_seed, wl.mlp_hidden)
        self.cache = dc.DistillCache(wl.layers, wl.kv_heads, wl.head_dim, cap, wl.budget, batch=wl.batch,
                                     q_heads=wl.q_heads, window=wl.window, mlp_hidden=wl.mlp_hidden,
                                     layernorm=wl.layernorm, alpha_mode=wl.alpha_mode, keep_features=True,
                                     seed=wl.policy_seed, scorer=scorer, global_tokens=True, engine=engine)
        self.cache.set_policy(self.blob)
        self.scorer = scorer
        R = wl.layers * wl.kv_heads
        alpha_mode = 1 if scorer == 1 else wl.alpha_mode
        self.oseqs = {b: oracle.OracleSeq(R, wl.head_dim, wl.group, wl.window, alpha_mode, cap) for b in self.seqs}
        self.step_idx = 0
        self.stats = {"attn_max_abs": 0.0, "evicted": 0}

    def rows_of(self, b):
        wl = self.wl
        return [(l * wl.batch + b) * wl.kv_heads + g for l in range(wl.layers) for g in range(wl.kv_heads)]

    def home(self, b):
        return b * self.wl.kv_heads

    def _dev(self, a):
        return self.torch.from_numpy(a.view(np.int16)).view(self.torch.bfloat16).cuda()

    def load_prompt(self):
        wl = self.wl
        k, v = synth.prompt_all(wl)
        self.cache.append(self._dev(k), self._dev(v))
        R = wl.layers * wl.kv_heads
        for b, o in self.oseqs.items():
            o.append(k[:, b].reshape(R, wl.prompt_len, wl.head_dim), v[:, b].reshape(R, wl.prompt_len, wl.head_dim))

    def _slice(self, which, r, n):
        return self.cache.buffer(which, r, 1)[0, :n].cpu().numpy()

    def step(self, check=True, budget=0):
        wl, dc = self.wl, self.dc
        s = self.step_idx
        q, kn, vn = synth.step_all(wl, s)
        out = self.cache.decode_step(self._dev(q), self._dev(kn), self._dev(vn)).cpu().numpy()
        self.cache.sync()
        n, _ = self.cache.length()
        R, G, d = wl.layers * wl.kv_heads, wl.group, wl.head_dim
        gpu_scores = {}
        for b, o in self.oseqs.items():
            res = o.step(q[:, b].reshape(R, G, d), kn[:, b].reshape(R, d), vn[:, b].reshape(R, d),
                         self.blob, wl.mlp_hidden, wl.layernorm)
            h = self.home(b)
            pos = self._slice(dc.BUF_POS, h, n)
            order = np.argsort(pos, kind="stable")
            assert np.array_equal(pos[order], res["pos"]), f"step {s} seq {b}: positions differ"
            sc = self._slice(dc.BUF_SCORE, h, n)[order]
            gpu_scores[b] = sc
            if not check:
                continue
            for j, r in enumerate(self.rows_of(b)):
                layer, _, g = wl.row_coords(r)
                ma, _ = check_attention(out[layer, b, g * G:(g + 1) * G], res["o"][j], f"step {s} row {r} attention")
                self.stats["attn_max_abs"] = max(self.stats["attn_max_abs"], ma)
            feat = self._slice(dc.BUF_FEAT, h, n)[order]
            for c, nm in enumerate(["alpha", "|v|", "sigma", "H", "pos"]):
                close_rel(feat[:, c], res["feat"][:, c], FEAT_RTOL, FEAT_FLOOR, f"step {s} seq {b} {nm}")
            if self.scorer == 2:  # sinks, then positions relative to the newest
                newest = res["pos"][-1]
                ref = np.where(res["pos"] < 4, np.float32(3e38), (res["pos"] - newest).astype(np.float32))
                assert np.array_equal(sc.astype(np.float32), ref.astype(np.float32)), f"step {s} seq {b} score"
            else:  # H2O ranks by the cumulative mass, the pooled alpha in cumulative mode
                ref = res["score"] if self.scorer == 0 else res["feat"][:, 0]
                close_rel(sc, ref, FEAT_RTOL, FEAT_FLOOR, f"step {s} seq {b} score")
        self.cache.evict(budget)
        self.cache.sync()
        B = budget if budget > 0 else wl.budget
        n2, _ = self.cache.length()
        assert n2 == min(n, B)
        self.stats["evicted"] += n - n2
        for b, o in self.oseqs.items():
            o.evict(B, gpu_scores[b])
            want = o.positions()
            for j, r in enumerate(self.rows_of(b)):
                pos = self._slice(dc.BUF_POS, r, n2)
                order = np.argsort(pos, kind="stable")
                assert np.array_equal(pos[order], want), f"step {s} row {r}: retained positions differ"
                K = self.cache.buffer(dc.BUF_K, r, 1)[0, :n2].view(self.torch.int16).cpu().numpy().view(np.uint16)
                V = self.cache.buffer(dc.BUF_V, r, 1)[0, :n2].view(self.torch.int16).cpu().numpy().view(np.uint16)
                ok, ov = o.kv_bits(j)
                assert np.array_equal(K[order], ok) and np.array_equal(V[order], ov), f"row {r}: K/V bytes differ"
            h = self.home(b)
            pos = self._slice(dc.BUF_POS, h, n2)
            order = np.argsort(pos, kind="stable")
            oS, oZ = o.window_sums_prior()
            close_rel(self._slice(dc.BUF_Z, h, n2)[order], oZ, FEAT_RTOL, FEAT_FLOOR, f"seq {b} window mass Z")
            close_rel(self._slice(dc.BUF_S, h, n2)[order], oS, FEAT_RTOL, FEAT_FLOOR, f"seq {b} window sum S")
        self.step_idx += 1
        return out
