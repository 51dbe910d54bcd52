"""GPU parity of wf_step, which runs the fused filter + sparse-attention
kernel (one thread-block cluster per (batch, head), tcgen05 tensor cores)
for bf16 / head_dim 128 / <= 32 query rows, against the fp64 oracle.

Same bars as the per-stage kernels: pyramid bit-exact, indices bit-exact on
planted inputs (every scale), bf16 outputs within max-abs 2e-2 and rel-L2
1e-2; unplanted inputs must give a valid Top-K at every scale."""
import numpy as np
import pytest
import torch

import oracle
from helpers import LibRun, assert_close_out, eps_valid, f64, make_layer, oracle_unit
from paper_2606_00724_gb300 import synth, wf

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)


def _check(w, batch, run, units):
    for u in units:
        b, h = divmod(u, w.heads)
        Q, K, V, Kg, Vg = (f64(t[b, h]) for t in (batch.Q, batch.K, batch.V, batch.Kg, batch.Vg))
        pyr, mu0, sets, O = oracle_unit(Q, K, V, Kg, Vg, w.levels, w.keep, True)
        assert np.array_equal(run.pyramid(u), pyr.astype(np.float64)), f"pyramid unit {u}"
        gsets = run.level_sets(u)
        for lev in range(w.levels, -1, -1):
            assert np.array_equal(gsets[lev], sets[lev]), f"unit {u} scale {lev}"
        assert np.array_equal(run.idx[u].cpu().numpy(), mu0), f"unit {u} mu0"
        assert_close_out(f64(run.O[b, h]), O, torch.bfloat16)


@pytest.mark.parametrize("cfg", ["c2", "c3", "c4", "c5"])
def test_step_full_size(cfg):
    w, batch = make_layer(cfg)
    run = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).step()
    wf.wf_workspace_status(run.ws_step)
    torch.cuda.synchronize()
    units = [0, 1, w.units // 2 + 3, w.units - 1]
    _check(w, batch, run, units)
    idx = run.idx.cpu().numpy()
    for u in range(w.units):
        assert np.array_equal(idx[u], batch.targets[u][0].cpu().numpy()), f"unit {u} planted"
    # Every unit's output against the oracle's attention over the kernel's
    # own indices (the selection itself is checked above).
    for u in range(w.units):
        b, h = divmod(u, w.heads)
        Q, K, V, Kg, Vg = (f64(t[b, h]) for t in (batch.Q, batch.K, batch.V, batch.Kg, batch.Vg))
        assert_close_out(f64(run.O[b, h]), oracle.sparse_attn(Q, K, V, idx[u], Kg, Vg), torch.bfloat16)


@pytest.mark.parametrize("cfg", ["c3", "c4"])
def test_step_unplanted_timing_inputs(cfg):
    # The distributions the benchmark times (c3: clustered keys, c4: keys with
    # a low-frequency drift), without planted margins: every sampled unit's
    # selection must be a valid Top-K at every scale (near-ties allow several
    # answers) and its output must match the oracle's attention over the
    # kernel's own indices.
    w, batch = make_layer(cfg, planted=False)
    run = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).step()
    wf.wf_workspace_status(run.ws_step)
    torch.cuda.synchronize()
    for u in [0, 5, w.units // 2 + 1, w.units - 1]:
        b, h = divmod(u, w.heads)
        Q, K, V, Kg, Vg = (f64(t[b, h]) for t in (batch.Q, batch.K, batch.V, batch.Kg, batch.Vg))
        pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), w.levels, True).astype(np.float64)
        assert np.array_equal(run.pyramid(u), pyr), f"pyramid unit {u}"
        gsets = run.level_sets(u)
        eps_valid(Q, pyr, K, w.n, w.levels, w.keep, gsets)
        idx = run.idx[u].cpu().numpy()
        assert np.array_equal(idx, gsets[0])
        assert_close_out(f64(run.O[b, h]), oracle.sparse_attn(Q, K, V, idx, Kg, Vg), torch.bfloat16)


def test_step_matches_per_stage_kernels():
    # Planted 8K layer: the fused kernel and the per-stage kernels select the
    # same indices and agree on the output.
    w, batch = make_layer("c2")
    a = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).run()
    b = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep)
    b.coeffs.copy_(a.coeffs)
    b.step(refresh=False)
    torch.cuda.synchronize()
    assert torch.equal(a.idx, b.idx)
    assert torch.equal(a.sets, b.sets)
    assert_close_out(f64(b.O), f64(a.O), torch.bfloat16)


def _rand(seed, B, H, n, q, ng, bshd=False):
    g = torch.Generator(device="cpu").manual_seed(seed)
    d = 128

    def r(rows):
        x = torch.randn(B, rows, H, d, generator=g) if bshd else torch.randn(B, H, rows, d, generator=g)
        x = x.to(torch.bfloat16).cuda()
        return x.transpose(1, 2) if bshd else x
    return r(q), r(n), r(n), (r(ng) if ng else None), (r(ng) if ng else None)


@pytest.mark.parametrize("B,H,n,q,ng,L,keep,bshd", [
    (1, 3, 4096, 32, 32, 3, [300, 150, 160, 170], False),          # cluster of 4, ragged tiles
    (2, 2, 2048, 7, 3, 2, [201, 101, 130], True),                  # trim, odd q, BSHD
    (1, 2, 1024, 1, 0, 1, [512, 256], False),                      # q = 1, no generation rows, L = 1
    (1, 1, 256, 32, 5, 4, [256, 128, 64, 32, 16], False),          # keep everything
    (1, 2, 512, 16, 1, 6, [1, 1, 1, 1, 1, 1, 1], False),           # k = 1, deep pyramid
    (1, 4, 65536, 32, 32, 5, [3000, 1500, 1600, 1700, 1800, 1900], False),  # large ragged schedule
])
def test_step_random_shapes(B, H, n, q, ng, L, keep, bshd):
    Q, K, V, Kg, Vg = _rand(n + q + L, B, H, n, q, ng, bshd)
    run = LibRun(Q, K, V, Kg, Vg, L, keep).step()
    wf.wf_workspace_status(run.ws_step)
    torch.cuda.synchronize()
    for u in range(B * H):
        b, h = divmod(u, H)
        Qn, Kn, Vn = f64(Q[b, h]), f64(K[b, h]), f64(V[b, h])
        Kgn = f64(Kg[b, h]) if ng else None
        Vgn = f64(Vg[b, h]) if ng else None
        pyr = oracle.haar_pyramid_spec32(Kn.astype(np.float32), L, True).astype(np.float64)
        assert np.array_equal(run.pyramid(u), pyr)
        gsets = run.level_sets(u)
        eps_valid(Qn, pyr, Kn, n, L, keep, gsets)
        idx = run.idx[u].cpu().numpy()
        assert np.array_equal(idx, gsets[0])
        assert np.all(np.diff(idx) > 0) and idx.min() >= 0 and idx.max() < n
        O = oracle.sparse_attn(Qn, Kn, Vn, idx, Kgn, Vgn)
        assert_close_out(f64(run.O[b, h]), O, torch.bfloat16)


@pytest.mark.parametrize("cfg", ["c2", "c3", "c4", "c5"])
def test_step_level0_schedule(cfg):
    # The token level as its own selection step (wf_level0_schedule): the
    # level-0 scan over raw keys keeps k of 2 keep[1] candidates.  Planted
    # ladder built for that schedule; full-size layer in the fused kernel
    # (at 128K the finest scales hold up to 7304 candidates: 64 keys a Top-K
    # thread).
    import dataclasses
    w0 = synth.WORKLOADS[cfg]
    keep = tuple(wf.wf_level0_schedule(w0.n, w0.levels, w0.k))
    assert keep[0] < 2 * keep[1]
    w = dataclasses.replace(w0, keep=keep, name=w0.name + "_level0")
    batch = synth.make_batch(w, planted=True, device="cuda", cfg=cfg)
    run = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, list(w.keep)).step()
    wf.wf_workspace_status(run.ws_step)
    torch.cuda.synchronize()
    _check(w, batch, run, [0, w.units // 2 + 1, w.units - 1])
    idx = run.idx.cpu().numpy()
    for u in range(w.units):
        assert np.array_equal(idx[u], batch.targets[u][0].cpu().numpy()), f"unit {u} planted"


@pytest.mark.parametrize("n,period,L,keep", [
    (8192, 64, 3, [512, 256, 300, 400]),            # groups of 128 equal keys: resolved by ranking
    (8192, 32, 3, [512, 256, 300, 400]),            # groups of 256: re-bucketed until only equal keys remain
    (32768, 64, 3, [2048, 1024, 1536, 2048]),       # 4096 keys a scale: 32 keys a Top-K thread
])
def test_step_exact_ties(n, period, L, keep):
    # K repeats one block of `period` tokens, so every scale's coefficient
    # rows, and with them the ranking keys, repeat exactly: the Top-K
    # boundary falls inside groups of bit-equal keys on both sides, and
    # Eq. 9's lower-position rule decides.  Indices must match the oracle
    # at every scale.
    g = torch.Generator(device="cpu").manual_seed(n + period)
    B, H, q, ng, d = 1, 2, 32, 8, 128

    def r(rows):
        return torch.randn(B, H, rows, d, generator=g).to(torch.bfloat16)
    Q, V, Kg, Vg = r(q).cuda(), r(n).cuda(), r(ng).cuda(), r(ng).cuda()
    K = r(period).repeat(1, 1, n // period, 1).contiguous().cuda()
    run = LibRun(Q, K, V, Kg, Vg, L, keep).step()
    wf.wf_workspace_status(run.ws_step)
    torch.cuda.synchronize()
    for u in range(B * H):
        Qn, Kn, Vn, Kgn, Vgn = (f64(t[0, u]) for t in (Q, K, V, Kg, Vg))
        pyr, mu0, sets, O = oracle_unit(Qn, Kn, Vn, Kgn, Vgn, L, keep, True)
        gsets = run.level_sets(u)
        for lev in range(L, -1, -1):
            assert np.array_equal(gsets[lev], sets[lev]), f"unit {u} scale {lev}"
        assert np.array_equal(run.idx[u].cpu().numpy(), mu0), f"unit {u} mu0"
        assert_close_out(f64(run.O[0, u]), O, torch.bfloat16)


@pytest.mark.parametrize("B,H,n,L,keep", [
    (1, 32, 8192, 3, [476, 442, 410, 819]),                # one unit a cluster: raised at the last key tile
    (2, 32, 32768, 4, [1024, 1024, 1024, 1024, 2048]),     # two units a cluster: raised mid-stream
    (1, 32, 32768, 4, [1024, 1024, 1024, 1024, 2048]),     # one unit on both warpgroups: raised at step 1
])
def test_step_raised_stabiliser(B, H, n, L, keep):
    # Generation row 0 of every unit gets logits of 55 to several hundred
    # (natural units) against every query row, far above the sparse keys'.
    # It sits in a later key tile of the last CTA of each cluster, so that
    # CTA's attention raises its stabiliser mid-stream (the accumulator and
    # the running sums are rescaled); the output must match the oracle's
    # attention over the kernel's own indices.
    Q, K, V, Kg, Vg = _rand(n + L + 77, B, H, n, 32, 32)
    # Every query row gets a component of 6 along one random direction per
    # unit, and generation row 0 points along it.
    g = torch.Generator(device="cpu").manual_seed(n + B)
    uvec = torch.randn(B, H, 128, generator=g, dtype=torch.float64)
    uvec = (uvec / uvec.norm(dim=-1, keepdim=True)).cuda()
    Q = (Q.double() + 6.0 * uvec[:, :, None, :]).to(torch.bfloat16)
    proj = torch.einsum("bhqd,bhd->bhq", Q.double(), uvec)
    lo = proj.min(dim=2).values
    assert torch.all(lo > 0.5)
    c = 55.0 * 128 ** 0.5 / lo
    Kg = Kg.clone()
    Kg[:, :, 0, :] = (c[..., None] * uvec).to(torch.bfloat16)
    run = LibRun(Q, K, V, Kg, Vg, L, keep).step()
    wf.wf_workspace_status(run.ws_step)
    torch.cuda.synchronize()
    for u in [0, 1, H - 1, B * H - 1]:
        b, h = divmod(u, H)
        Qn, Kn, Vn, Kgn, Vgn = (f64(t[b, h]) for t in (Q, K, V, Kg, Vg))
        s = Qn @ Kgn[0] / np.sqrt(128)
        assert s.min() >= 54.0
        idx = run.idx[u].cpu().numpy()
        pyr = oracle.haar_pyramid_spec32(Kn.astype(np.float32), L, True).astype(np.float64)
        eps_valid(Qn, pyr, Kn, n, L, keep, run.level_sets(u))
        assert_close_out(f64(run.O[b, h]), oracle.sparse_attn(Qn, Kn, Vn, idx, Kgn, Vgn), torch.bfloat16)
