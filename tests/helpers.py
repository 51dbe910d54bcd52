"""Shared helpers for the GPU parity tests: run libwf on a batch, run the
oracle on chosen units, and compare."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2606_00724_gb300 import synth
from paper_2606_00724_gb300 import wf


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu", torch.float64).numpy()


class LibRun:
    """Buffers and outputs of one libwf pass over a [B, H, ...] layer."""

    def __init__(self, Q, K, V, Kg, Vg, L, keep, want_sets=True):
        dev = K.device
        self.Q, self.K, self.V, self.Kg, self.Vg = Q, K, V, Kg, Vg
        self.L, self.keep = L, [int(x) for x in keep]
        B, H = K.shape[0], K.shape[1]
        self.coeffs = torch.empty(wf.wf_coeffs_bytes(K, L), dtype=torch.uint8, device=dev)
        ws_bytes = max(wf.wf_filter_workspace_bytes(Q, K, L, self.keep),
                       wf.wf_attn_workspace_bytes(Q, self.keep[0], Kg.shape[2] if Kg is not None else 0))
        self.ws = torch.zeros(ws_bytes, dtype=torch.uint8, device=dev)  # status word zeroed once
        self.idx = torch.empty(B * H, self.keep[0], dtype=torch.int32, device=dev)
        self.sets = torch.empty(B * H, sum(self.keep), dtype=torch.int32, device=dev) if want_sets else None
        self.O = torch.empty_like(Q)

    def dwt(self):
        wf.wf_dwt_build(self.K, self.L, self.coeffs)
        return self

    def filter(self):
        wf.wf_filter(self.Q, self.coeffs, self.K, self.L, self.keep, self.idx, self.ws, self.sets)
        wf.wf_workspace_status(self.ws)  # raises if a bounded device wait gave up
        return self

    def attn(self, idx=None, scale=0.0):
        idx = self.idx if idx is None else idx
        wf.wf_sparse_attn(self.Q, self.K, self.V, idx, idx.shape[1], self.Kg, self.Vg, self.O, self.ws, scale)
        return self

    def run(self):
        return self.dwt().filter().attn()

    def step(self, refresh=True):
        """One wf_step (fused kernel where it applies), with level sets."""
        if not hasattr(self, "ws_step"):
            ng = self.Kg.shape[2] if self.Kg is not None else 0
            self.ws_step = torch.zeros(wf.wf_step_workspace_bytes(self.Q, self.K, self.L, self.keep, ng),
                                       dtype=torch.uint8, device=self.K.device)
        wf.wf_step(self.Q, self.K, self.V, self.Kg, self.Vg, self.coeffs, refresh, self.L, self.keep, self.idx,
                   self.O, self.ws_step, level_sets=self.sets)
        return self

    def pyramid(self, u: int) -> np.ndarray:
        """Stored pyramid rows of unit u as float64."""
        B, H, n, d = self.K.shape
        rows = n - (n >> self.L)
        dt = self.K.dtype
        c = self.coeffs.view(dt).view(B * H, rows, d)[u]
        return f64(c)

    def level_sets(self, u: int) -> dict:
        return oracle.split_level_sets(self.sets[u].cpu().numpy(), self.L, self.keep)


def unit_arrays(batch_tensors, u: int, H: int):
    b, h = divmod(u, H)
    return [f64(t[b, h]) if t is not None else None for t in batch_tensors]


def oracle_unit(Q, K, V, Kg, Vg, L, keep, store_bf16):
    """Oracle outputs for one unit: stored pyramid, mu0, level sets, O."""
    pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), L, store_bf16)
    mu0, sets = oracle.filter(Q, pyr, K, K.shape[0], L, np.array(keep), want_sets=True)
    O = oracle.sparse_attn(Q, K, V, mu0, Kg, Vg)
    return pyr, mu0, sets, O


def assert_close_out(got: np.ndarray, want: np.ndarray, dtype: torch.dtype):
    """Output tolerances: fp32 max-abs 1e-5; bf16 max-abs 2e-2 and rel-L2 1e-2."""
    err = np.abs(got - want)
    if dtype == torch.float32:
        assert err.max() <= 1e-5, f"max-abs {err.max():.3g} > 1e-5"
    else:
        rel = np.linalg.norm(got - want) / max(np.linalg.norm(want), 1e-30)
        assert err.max() <= 2e-2, f"max-abs {err.max():.3g} > 2e-2"
        assert rel <= 1e-2, f"rel-L2 {rel:.3g} > 1e-2"


def eps_valid(Q, pyr64, K64, n, L, keep, gpu_sets: dict, rel_eps=1e-5):
    """Check a GPU selection is a valid Top-K at every scale when near-ties
    make several answers correct: re-score the GPU's own candidates in fp64
    and require min W over the kept set >= max W over the rest - eps."""
    cand = np.arange(n >> L)
    for b in range(L, 0, -1):
        rows = oracle.level(pyr64, n, b)[cand]
        W = oracle.skim_weights(Q, rows)
        kept = np.isin(cand, gpu_sets[b])
        assert kept.sum() == keep[b]
        if kept.sum() < cand.size:
            assert W[kept].min() >= W[~kept].max() - rel_eps * W.max(), f"scale {b} not a valid top-k"
        cand = np.stack([2 * gpu_sets[b], 2 * gpu_sets[b] + 1], 1).reshape(-1)
    if keep[0] < cand.size:
        W = oracle.skim_weights(Q, K64[cand])
        kept = np.isin(cand, gpu_sets[0])
        assert kept.sum() == keep[0]
        assert W[kept].min() >= W[~kept].max() - rel_eps * W.max(), "level-0 trim not a valid top-k"
    else:
        assert np.array_equal(np.sort(cand), gpu_sets[0])


def make_layer(cfg: str, planted=True, device="cuda", units=None, layer=0):
    w = synth.WORKLOADS[cfg]
    return w, synth.make_batch(w, layer=layer, planted=planted, device=device, cfg=cfg, units=units)
