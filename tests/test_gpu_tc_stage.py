"""GPU parity of the tensor-core per-stage kernels (bf16, head_dim 128):
the tcgen05 skim inside wf_filter and the tcgen05 split attention inside
wf_sparse_attn, on shapes the workloads do not reach: query blocks that are
not a multiple of 32 rows (1, 17, 40, and 3 grouped heads of 20), sparse
key counts that leave ragged 128-key splits, no generation rows, BSHD
strides, a non-default attention scale.  Indices bit-exact against the
oracle on planted inputs; outputs within the bf16 bound."""
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


def _workload(q, group, n=4096, L=3, k=512, ng=32, heads=2):
    w = dataclasses.replace(synth.WORKLOADS["g1"], batch=1, heads=heads, group=group, q=q, n=n, levels=L, ng=ng)
    return dataclasses.replace(w, keep=tuple(int(x) for x in oracle.default_schedule(n, L, k)), name="tc_variant")


@pytest.mark.parametrize("q,group,k,ng", [(1, 1, 512, 32), (17, 1, 300, 0), (40, 1, 640, 7), (20, 3, 512, 32),
                                          (32, 8, 257, 1)])
def test_tc_filter_and_attention(q, group, k, ng):
    w = _workload(q, group, k=k, ng=ng)
    batch = synth.make_batch(w, planted=True, device="cuda", cfg="g1")
    Kg = batch.Kg if ng else None
    Vg = batch.Vg if ng else None
    run = LibRun(batch.Q, batch.K, batch.V, Kg, Vg, w.levels, w.keep).run()
    wf.wf_workspace_status(run.ws)
    torch.cuda.synchronize()
    G = w.group
    for u in range(w.units):
        b, h = divmod(u, w.heads)
        Qh = f64(batch.Q[b, h * G:(h + 1) * G])
        K, V = f64(batch.K[b, h]), f64(batch.V[b, h])
        pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), w.levels, True)
        mu0, sets = oracle.filter_gqa(Qh, pyr, K, w.n, w.levels, np.array(w.keep), want_sets=True)
        gsets = run.level_sets(u)
        for lev in range(w.levels, -1, -1):
            assert np.array_equal(gsets[lev], sets[lev]), f"unit {u} scale {lev}"
            assert np.array_equal(gsets[lev], batch.targets[u][lev].cpu().numpy()), f"unit {u} planted {lev}"
        kg = f64(batch.Kg[b, h]) if ng else None
        vg = f64(batch.Vg[b, h]) if ng else None
        O = oracle.sparse_attn_gqa(Qh, K, V, mu0, kg, vg)
        assert_close_out(f64(run.O[b, h * G:(h + 1) * G]), O, torch.bfloat16)


def test_tc_attention_bshd_and_scale():
    # Random (unsorted) index lists, BSHD caches, an explicit scale.
    B, H, n, d, q, k, ng = 2, 3, 2048, 128, 24, 333, 5
    g = torch.Generator(device="cpu").manual_seed(3)
    bshd = lambda rows, heads=H: torch.randn(B, rows, heads, d, generator=g).to(torch.bfloat16).cuda().transpose(1, 2)
    Q, K, V, Kg, Vg = bshd(q), bshd(n), bshd(n), bshd(ng), bshd(ng)
    idx = torch.stack([torch.randperm(n, generator=g)[:k] for _ in range(B * H)]).to(torch.int32).cuda()
    O = torch.empty(B, H, q, d, dtype=torch.bfloat16, device="cuda")
    ws = torch.zeros(wf.wf_attn_workspace_bytes(O, k, ng), dtype=torch.uint8, device="cuda")
    scale = 0.05
    wf.wf_sparse_attn(Q, K, V, idx, k, Kg, Vg, O, ws, scale)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    for u in range(B * H):
        b, h = divmod(u, H)
        Ks = np.concatenate([f64(K[b, h])[idx[u].cpu().numpy()], f64(Kg[b, h])])
        Vs = np.concatenate([f64(V[b, h])[idx[u].cpu().numpy()], f64(Vg[b, h])])
        s = f64(Q[b, h]) @ Ks.T * scale
        p = np.exp(s - s.max(axis=1, keepdims=True))
        want = (p / p.sum(axis=1, keepdims=True)) @ Vs
        assert_close_out(f64(O[b, h]), want, torch.bfloat16)
