"""GPU parity of grouped-query attention (GQA): one selection per key head
from the stacked query rows of its G query heads, then every query head
attends over its key head's selected rows.

Bars: indices bit-exact on planted inputs at every scale (against the planted
answer and the oracle), outputs within the dtype's bound (fp32 max-abs 1e-5;
bf16 max-abs 2e-2, rel-L2 1e-2); wf_step gives what wf_filter +
wf_sparse_attn give."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from helpers import LibRun, assert_close_out, f64
from paper_2606_00724_gb300 import synth, wf

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)


def _workload(base, k=None, **kw):
    w = dataclasses.replace(synth.WORKLOADS[base], **kw)
    keep = oracle.default_schedule(w.n, w.levels, w.k if k is None else k)
    return dataclasses.replace(w, keep=tuple(int(x) for x in keep), name=w.name + "_variant")


def _check_units(w, batch, run, units, dtype):
    G = w.group
    for u in units:
        b, h = divmod(u, w.heads)
        Qh = f64(batch.Q[b, h * G:(h + 1) * G])
        K, V, Kg, Vg = (f64(t[b, h]) for t in (batch.K, batch.V, batch.Kg, batch.Vg))
        pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), w.levels, dtype == torch.bfloat16)
        assert np.array_equal(run.pyramid(u), pyr.astype(np.float64)), f"pyramid unit {u}"
        mu0, sets = oracle.filter_gqa(Qh, pyr, K, w.n, w.levels, np.array(w.keep), want_sets=True)
        if run.sets is not None:
            gsets = run.level_sets(u)
            for lev in range(w.levels, -1, -1):
                assert np.array_equal(gsets[lev], sets[lev]), f"unit {u} scale {lev}"
                assert np.array_equal(gsets[lev], batch.targets[u][lev].cpu().numpy()), f"unit {u} planted {lev}"
        assert np.array_equal(run.idx[u].cpu().numpy(), mu0), f"unit {u} mu0"
        O = oracle.sparse_attn_gqa(Qh, K, V, mu0, Kg, Vg)
        assert_close_out(f64(run.O[b, h * G:(h + 1) * G]), O, dtype)


@pytest.mark.parametrize("base,kw,dtype", [
    # Dream-7B grouping (7 query heads per key head), shorter context.
    ("g1", dict(batch=2, heads=2, n=4096, levels=3, k=512), torch.bfloat16),
    # Two heads per key head, head_dim 64, fp32 (the fp32 bar: max-abs 1e-5).
    ("c1", dict(heads=2, group=2), torch.float32),
    # Eight heads per key head: 8 x 32 = 256 query rows per key head (the limit).
    ("g1", dict(batch=1, heads=1, group=8, n=2048, levels=2, k=256), torch.bfloat16),
])
def test_gqa_per_stage(base, kw, dtype):
    w = _workload(base, **kw)
    cfg = base
    batch = synth.make_batch(w, planted=True, device="cuda", cfg=cfg)
    assert batch.Q.dtype == dtype and batch.Q.shape[1] == w.heads * w.group
    run = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).run()
    torch.cuda.synchronize()
    _check_units(w, batch, run, range(w.units), dtype)
    # wf_step (the grouped filter kernel for bf16, else the per-stage path):
    # same indices, same output.
    step = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep)
    step.step()
    torch.cuda.synchronize()
    assert torch.equal(step.idx, run.idx)
    assert torch.equal(step.sets, run.sets)
    assert torch.equal(step.O, run.O)


def test_gqa_dream_shape_sampled_units():
    # The full Dream-shaped layer (B8, 28 query heads on 4 key heads, 32K
    # context): wf_step on the whole layer; sampled units against the oracle.
    w = synth.WORKLOADS["g1"]
    units = [0, 13, w.units - 1]
    batch = synth.make_batch(w, planted=True, device="cuda", cfg="g1", units=units)
    run = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).dwt().step(refresh=False)
    torch.cuda.synchronize()
    _check_units(w, batch, run, units, torch.bfloat16)


def test_gqa_attention_equals_repeated_key_heads():
    # The head mapping of the grouped attention (query head h G + g reads key
    # head h and its index row) against the ungrouped call on key heads
    # repeated G times, with the same selection.  The grouped call (96 query
    # rows a key head) runs the kernel with the query rows on the TMEM lanes,
    # the ungrouped one (32 rows) the kernel with the keys on the lanes: the
    # two outputs agree within the bf16 bound, and the grouped one matches the
    # oracle unit by unit.
    w = _workload("g1", batch=2, heads=2, group=3, n=2048, levels=2, k=256)
    batch = synth.make_batch(w, planted=True, device="cuda", cfg="g1")
    G = w.group
    grouped = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).run()
    rep = lambda t: t.repeat_interleave(G, dim=1).contiguous()
    K1, V1, Kg1, Vg1 = rep(batch.K), rep(batch.V), rep(batch.Kg), rep(batch.Vg)
    idx1 = grouped.idx.repeat_interleave(G, dim=0).contiguous()
    O1 = torch.empty_like(batch.Q)
    ws = torch.zeros(wf.wf_attn_workspace_bytes(batch.Q, w.k, w.ng), dtype=torch.uint8, device="cuda")
    wf.wf_sparse_attn(batch.Q, K1, V1, idx1, w.k, Kg1, Vg1, O1, ws)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    assert_close_out(f64(O1), f64(grouped.O), torch.bfloat16)
    _check_units(w, batch, grouped, range(w.units), torch.bfloat16)


@pytest.mark.parametrize("kw,units,hot,cold", [
    (dict(), [0, 17, 31], 0.0, False),                                    # the Dream-shaped layer: clusters of 4, 4 tiles a scale
    (dict(batch=1, heads=4, n=8192, levels=3, k=819), [0, 3], 0.0, False),  # clusters of 8, one tile a scale, level-0 trim
    (dict(batch=1, heads=4, n=8192, levels=3, k=819), [0, 3], 80.0, False),  # one query row 80x: other rows' terms flush
    (dict(batch=1, heads=4, n=8192, levels=3, k=819), [0, 3], 0.0, True),   # key rows far below every query: tiny W
])
def test_gqa_step_unplanted_valid_topk(kw, units, hot, cold):
    # wf_step's grouped filter kernel on unplanted inputs: at every scale the
    # selection must be a valid Top-K of W summed over the key head's stacked
    # query rows (near-ties allow several answers), and the output must match
    # the oracle's grouped attention over the kernel's own indices.  With
    # `hot`, row 0 of every unit's first query head is scaled so that its
    # logits lie hundreds of units above the chunk's other rows: their
    # exponentials against the chunk's largest logit flush to zero, and the
    # filter must sum those columns against their own maxima.  With `cold`,
    # some candidates' W are tiny and their keys are taken shifted.
    from helpers import eps_valid
    w = _workload("g1", **kw) if kw else synth.WORKLOADS["g1"]
    batch = synth.make_batch(w, planted=False, device="cuda", cfg="g1", units=units)
    if hot:
        Q = batch.Q.clone()
        Q[:, ::w.group, 0, :] = (Q[:, ::w.group, 0, :].float() * hot).to(Q.dtype)
        batch = dataclasses.replace(batch, Q=Q)
    if cold:
        # Every query row of a unit gets a component of 6 along one direction
        # u; 256 key tokens point along -u with logits near -80 for every
        # query row, so their candidates' W lie far below 2^-96.
        g = torch.Generator(device="cpu").manual_seed(5)
        u = torch.randn(w.batch, w.heads, w.head_dim, generator=g, dtype=torch.float64)
        u = (u / u.norm(dim=-1, keepdim=True)).cuda()
        ug = u.repeat_interleave(w.group, dim=1)
        Q = (batch.Q.double() + 6.0 * ug[:, :, None, :]).to(batch.Q.dtype)
        K = batch.K.clone()
        K[:, :, 2048:2304, :] = (-(80.0 / 6.0) * 128 ** 0.5 * u[:, :, None, :]).to(K.dtype)
        batch = dataclasses.replace(batch, Q=Q, K=K)
    run = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).dwt().step(refresh=False)
    wf.wf_workspace_status(run.ws_step)
    torch.cuda.synchronize()
    G = w.group
    for u in units:
        b, h = divmod(u, w.heads)
        Qh = f64(batch.Q[b, h * G:(h + 1) * G])
        K, V, Kg, Vg = (f64(t[b, h]) for t in (batch.K, batch.V, batch.Kg, batch.Vg))
        pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), w.levels, True).astype(np.float64)
        gsets = run.level_sets(u)
        eps_valid(Qh.reshape(-1, Qh.shape[-1]), pyr, K, w.n, w.levels, list(w.keep), gsets)
        idx = run.idx[u].cpu().numpy()
        assert np.array_equal(idx, gsets[0])
        O = oracle.sparse_attn_gqa(Qh, K, V, idx, Kg, Vg)
        assert_close_out(f64(run.O[b, h * G:(h + 1) * G]), O, torch.bfloat16)


def test_gqa_attention_raised_stabiliser():
    # The attention with the query rows on the TMEM lanes raises a row's
    # stabiliser only when a tile's max exceeds it by more than 8 (log2
    # units), and then rescales the partial O and row sum.  16 key units of
    # 17 key tiles give CTAs of two consecutive tiles; every query row has a
    # component of 4 along one direction u, and the keys of the odd tiles
    # get one along u too, so that an odd tile's max lies about 5 (tiles
    # 1, 5, 9, 13: the stabiliser is kept, P up to 2^5) or about 20 (tiles
    # 3, 7, 11, 15: raised, O rescaled) above the even tile's before it.
    B, H, G, qs, n, d, k, ng = 2, 8, 7, 32, 8192, 128, 2048, 32
    gen = torch.Generator(device="cpu").manual_seed(11)
    u = torch.randn(B, H, d, generator=gen, dtype=torch.float64)
    u = u / u.norm(dim=-1, keepdim=True)
    Q = torch.randn(B, H * G, qs, d, generator=gen, dtype=torch.float64)
    Q = Q + 4.0 * u.repeat_interleave(G, dim=1)[:, :, None, :]
    K = torch.randn(B, H, n, d, generator=gen, dtype=torch.float64)
    V = torch.randn(B, H, n, d, generator=gen, dtype=torch.float64)
    Kg = torch.randn(B, H, ng, d, generator=gen, dtype=torch.float64)
    Vg = torch.randn(B, H, ng, d, generator=gen, dtype=torch.float64)
    idx = torch.stack([torch.randperm(n, generator=gen)[:k].sort().values for _ in range(B * H)])
    amp = torch.zeros(k, dtype=torch.float64)
    tile = torch.arange(k) // 128
    amp[tile % 4 == 1] = 10.0
    amp[tile % 4 == 3] = 40.0
    for un in range(B * H):
        b, h = divmod(un, H)
        K[b, h, idx[un]] += amp[:, None] * u[b, h][None, :]
    bf = lambda t: t.to(torch.bfloat16).cuda().contiguous()
    Qd, Kd, Vd, Kgd, Vgd = bf(Q), bf(K), bf(V), bf(Kg), bf(Vg)
    idx_d = idx.to(torch.int32).cuda()
    O = torch.empty_like(Qd)
    ws = torch.zeros(wf.wf_attn_workspace_bytes(Qd, k, ng), dtype=torch.uint8, device="cuda")
    wf.wf_sparse_attn(Qd, Kd, Vd, idx_d, k, Kgd, Vgd, O, ws)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    for un in range(B * H):
        b, h = divmod(un, H)
        Qh = f64(Qd[b, h * G:(h + 1) * G])
        want = oracle.sparse_attn_gqa(Qh, f64(Kd[b, h]), f64(Vd[b, h]), idx[un].numpy(), f64(Kgd[b, h]),
                                      f64(Vgd[b, h]))
        assert_close_out(f64(O[b, h * G:(h + 1) * G]), want, torch.bfloat16)
