"""Seeded synthetic workloads for the WaveFilter hot path.

The paper evaluates on LongBench and RULER with LLaDA-8B-Instruct and
Dream-v0-Base-7B (Section 4.1); none of those is available here, so these
generators stand in for them with inputs of the same shapes (32 heads x 128
head dims, 8K-128K prompt tokens, a 32-row denoising block) and with the
structures that make the filter's job non-trivial: needles, RoPE-like
positional rotations, piecewise-constant topic clusters, slow drift.

This module holds none of the method's arithmetic: it draws tensors and,
when asked, plants a known answer ("planted ladder") by adding a bonus
direction to chosen token blocks.  The kept counts per scale are explicit
inputs of each workload.  Both the oracle side and the CUDA side of the tests
consume its outputs, so the two sides always see the same inputs.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    heads: int
    head_dim: int
    n: int            # prompt tokens |I_p|
    q: int            # query rows of the denoising block |I~|
    ng: int           # generation rows |I_g| appended to the sparse set
    levels: int       # DWT scale B
    keep: tuple       # keep[b] for b = 0..L (keep[0] = k tokens)
    dtype: str        # "f32" or "bf16"
    kind: str
    layers: int = 1
    refresh_every: int = 0
    extra: dict = field(default_factory=dict)
    group: int = 1    # query heads per KV head (grouped-query attention); `heads` counts KV heads

    @property
    def k(self) -> int:
        return int(self.keep[0])

    @property
    def q_heads(self) -> int:
        return self.heads * self.group

    @property
    def units(self) -> int:
        return self.batch * self.heads


# keep[] = kept coefficient counts per scale b (index b), keep[0] = k.  They
# are the default schedule m = (k/n)^(1/L) evaluated for each shape, stated
# here as data.
WORKLOADS = {
    "c1": Workload("c1_tiny_fp32_n1k", 1, 4, 64, 1024, 32, 32, 2, (128, 64, 91), "f32", "needles",
                   extra={"needles": 8}),
    "c2": Workload("c2_llada_n8k", 1, 32, 128, 8192, 32, 32, 3, (819, 410, 442, 476), "bf16", "rope_spans",
                   extra={"spans": 32, "span_len": 16}),
    "c3": Workload("c3_llada_n32k_b2", 2, 32, 128, 32768, 32, 32, 4, (2048, 1024, 1024, 1024, 1024), "bf16",
                   "clusters", extra={"centroids": 64, "seg_min": 256, "seg_max": 2048, "needle_frac": 0.001,
                                      "gap_growth": 2.0 ** 0.5}),
    "c4": Workload("c4_llada_n128k", 1, 32, 128, 131072, 32, 32, 5, (4096, 2048, 2048, 2048, 2048, 2048), "bf16",
                   "drift", extra={"period": 4096, "needles": 128, "gap_growth": 2.0 ** 0.5}),
    "c5": Workload("c5_llada_32layer_n32k_b4", 4, 32, 128, 32768, 32, 32, 4, (1638, 819, 868, 917, 969), "bf16",
                   "iid", layers=32, refresh_every=8),
    # Grouped-query attention with the Dream-7B head layout (28 query heads
    # sharing 4 KV heads, head_dim 128): one selection per KV head.
    "g1": Workload("g1_dream_gqa_n32k_b8", 8, 4, 128, 32768, 32, 32, 4, (2048, 1024, 1024, 1024, 1024), "bf16",
                   "clusters", extra={"centroids": 64, "seg_min": 256, "seg_max": 2048, "needle_frac": 0.001,
                                      "gap_growth": 2.0 ** 0.5}, group=7),
}

CONFIG_NUMBER = {"c1": 1, "c2": 2, "c3": 3, "c4": 4, "c5": 5, "g1": 6}

# Planted ladder constants: every query gets a component PLANT_C along the
# unit direction u; each chosen scale-b block gets a bonus that lifts its
# scale-b logit by PLANT_GAP * gap_growth^b for every query.  Workloads whose
# keys carry low-frequency structure (clusters, drift) see a natural logit
# spread that grows like 2^(b/2) with the scale, so their gap grows with it.
PLANT_C = 2.0
PLANT_GAP = 8.0


def unit_seed(cfg: str, layer: int, b: int, h: int, salt: int = 0) -> int:
    base = 1000 * CONFIG_NUMBER.get(cfg, 9) + layer
    return (base * 1_000_003 + b * 10_007 + h * 101 + salt * 7_919) % (2**62)


@dataclass
class Unit:
    """One (batch, KV head) unit, fp32 tensors before storage rounding."""
    Q: torch.Tensor       # [group * q, d]: the q rows of each query head of the group, head after head
    K: torch.Tensor       # [n, d]
    V: torch.Tensor       # [n, d]
    Kg: torch.Tensor      # [ng, d]
    Vg: torch.Tensor      # [ng, d]
    targets: dict | None  # {b: planted J_b (ascending int64)}, key 0 = planted mu0
    needles: torch.Tensor  # token positions of planted needles


def _needle_keys(Q: torch.Tensor, rows: torch.Tensor, d: int) -> torch.Tensor:
    # A needle key is 4 sqrt(d) times the unit direction of one query row.
    qn = Q[rows]
    return 4.0 * math.sqrt(d) * qn / qn.norm(dim=1, keepdim=True)


def _rope(x: torch.Tensor, pos: torch.Tensor, omega: torch.Tensor) -> torch.Tensor:
    # Rotate channel pairs (2i, 2i+1) by angle pos * omega_i.
    ang = pos[:, None].to(torch.float64) * omega[None, :].to(torch.float64)
    c = torch.cos(ang).to(x.dtype)
    s = torch.sin(ang).to(x.dtype)
    x0 = x[:, 0::2]
    x1 = x[:, 1::2]
    out = torch.empty_like(x)
    out[:, 0::2] = x0 * c - x1 * s
    out[:, 1::2] = x0 * s + x1 * c
    return out


def make_unit(w: Workload, b: int, h: int, layer: int = 0, planted: bool = True,
              device: str | torch.device = "cpu", cfg: str | None = None) -> Unit:
    cfg = cfg or next(key for key, val in WORKLOADS.items() if val == w)
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(unit_seed(cfg, layer, b, h))
    d, n, q, ng = w.head_dim, w.n, w.q, w.ng
    qr = q * w.group  # query rows of the unit
    f32 = torch.float32

    def randn(*shape):
        return torch.randn(*shape, generator=g, device=dev, dtype=f32)

    def randint(lo, hi, shape):
        return torch.randint(lo, hi, shape, generator=g, device=dev)

    Q = randn(qr, d)
    V = randn(n, d)
    Kg = randn(ng, d)
    Vg = randn(ng, d)
    needles = torch.zeros(0, dtype=torch.int64, device=dev)
    if w.kind == "needles" or w.kind == "iid":
        K = randn(n, d)
    elif w.kind == "rope_spans":
        K = randn(n, d)
        omega = (10000.0 ** (-2.0 * torch.arange(d // 2, device=dev, dtype=torch.float64) / d)) * (
            0.5 + torch.rand(d // 2, generator=g, device=dev, dtype=torch.float64))
        K = _rope(K, torch.arange(n, device=dev), omega)
        Q = _rope(Q, torch.arange(n, n + q, device=dev).repeat(w.group), omega)
        Kg = _rope(Kg, torch.arange(n, n + ng, device=dev), omega)
    elif w.kind == "clusters":
        cent = randn(w.extra["centroids"], d)
        lo, hi = w.extra["seg_min"], w.extra["seg_max"]
        ids = torch.empty(n, dtype=torch.int64, device=dev)
        t = 0
        while t < n:
            ln = int(randint(lo, hi + 1, (1,)).item())
            ids[t: t + ln] = int(randint(0, cent.shape[0], (1,)).item())
            t += ln
        K = cent[ids] + 0.5 * randn(n, d)
    elif w.kind == "drift":
        period = w.extra["period"]
        phik = 2 * math.pi * torch.rand(d, generator=g, device=dev, dtype=f32)
        phiv = 2 * math.pi * torch.rand(d, generator=g, device=dev, dtype=f32)
        tt = torch.arange(n, device=dev, dtype=torch.float64)[:, None] * (2 * math.pi / period)
        K = randn(n, d) + torch.sin(tt + phik[None, :].double()).to(f32)
        V = V + torch.sin(tt + phiv[None, :].double()).to(f32)
    else:
        raise ValueError(w.kind)

    # Needles.
    if w.kind == "needles" or w.kind == "drift":
        cnt = w.extra["needles"]
        needles = torch.randperm(n, generator=g, device=dev)[:cnt].sort().values
    elif w.kind == "clusters":
        cnt = int(round(w.extra["needle_frac"] * n))
        needles = torch.randperm(n, generator=g, device=dev)[:cnt].sort().values
    elif w.kind == "rope_spans":
        span, cnt = w.extra["span_len"], w.extra["spans"]
        starts = torch.randperm(n // span, generator=g, device=dev)[:cnt] * span
        starts = starts + randint(0, span // 2, (cnt,))
        starts = starts.clamp(max=n - span)
        needles = (starts[:, None] + torch.arange(span, device=dev)[None, :]).reshape(-1).unique()
    if needles.numel():
        rows = randint(0, qr, (needles.numel(),))
        K[needles] = _needle_keys(Q, rows, d)

    targets = None
    if planted:
        targets = _plant(w, g, dev, Q, K, Kg, needles)
    return Unit(Q, K, V, Kg, Vg, targets, needles)


def _plant(w: Workload, g: torch.Generator, dev, Q, K, Kg, needles) -> dict:
    """Planted ladder: pick target sets top-down and lift them along u.

    Every query's component along a random unit direction u is set to
    PLANT_C.  Scale L: keep[L] blocks are chosen (blocks holding needles
    first, the rest at random) and each token of a chosen block gets
    +beta_L along u.  Finer scales b = L-1..1 and the optional level-0 trim:
    the candidates are the two children of every block chosen one scale up;
    keep[b] of them are chosen, needle blocks first, then at most one child
    per parent while the count allows.  A chosen child gets +beta_b and, when
    its sibling is not chosen, the sibling gets -beta_b, so the parent's
    coefficient (the sum of its children) is unchanged and the bonuses of
    finer scales do not leak into coarser ones.  beta_b = G_b sqrt(d) /
    (PLANT_C 2^(b/2)) lifts a scale-b coefficient's logit by
    G_b = PLANT_GAP * gap_growth^b for every query.  The generation rows get
    the whole bonus of a chosen token so they stay competitive in the final
    attention.
    """
    d, n, L = w.head_dim, w.n, w.levels
    keep = [int(x) for x in w.keep]
    u = torch.randn(d, generator=g, device=dev, dtype=torch.float64)
    u = u / u.norm()
    uf = u.to(torch.float32)
    Q -= (Q.double() @ u)[:, None].to(torch.float32) * uf[None, :]
    Q += PLANT_C * uf[None, :]
    bonus = torch.zeros(n, dtype=torch.float64, device=dev)
    cand = torch.arange(n >> L, device=dev)
    targets = {}
    total = 0.0
    for b in range(L, -1, -1):
        if b == 0 and keep[0] >= cand.numel():
            targets[0] = cand.clone()
            break
        kb = keep[b]
        forced = torch.unique(needles >> b) if needles.numel() else needles
        is_forced = torch.isin(cand, forced)
        nf = int(is_forced.sum())
        if nf > kb:
            raise ValueError(f"{w.name}: {nf} needle blocks exceed keep[{b}]={kb}")
        chosen_mask = is_forced.clone()
        if b == L:
            rest = torch.nonzero(~is_forced).reshape(-1)
            chosen_mask[rest[torch.randperm(rest.numel(), generator=g, device=dev)[: kb - nf]]] = True
        else:
            cm = chosen_mask.view(-1, 2)
            free = torch.nonzero(~cm.any(dim=1)).reshape(-1)
            free = free[torch.randperm(free.numel(), generator=g, device=dev)]
            first = free[: kb - nf]
            side = torch.randint(0, 2, (first.numel(),), generator=g, device=dev)
            cm[first, side] = True
            extra = kb - nf - first.numel()
            if extra > 0:
                rest = torch.nonzero(~chosen_mask).reshape(-1)
                chosen_mask[rest[torch.randperm(rest.numel(), generator=g, device=dev)[:extra]]] = True
        chosen = cand[chosen_mask]
        targets[b] = chosen
        gap = PLANT_GAP * w.extra.get("gap_growth", 1.0) ** b
        beta = gap * math.sqrt(d) / (PLANT_C * 2.0 ** (b / 2.0))
        total += beta
        val = torch.zeros(cand.numel(), dtype=torch.float64, device=dev)
        val[chosen_mask] = beta
        if b < L:
            cm = chosen_mask.view(-1, 2)
            lone = (cm.sum(dim=1) == 1)[:, None] & ~cm
            val.view(-1, 2)[lone] = -beta
        tok = (cand[:, None] << b) + torch.arange(1 << b, device=dev)[None, :]
        bonus[tok.reshape(-1)] += val[:, None].expand(-1, 1 << b).reshape(-1)
        cand = torch.stack([2 * chosen, 2 * chosen + 1], dim=1).reshape(-1)
    K += (bonus[:, None] * u[None, :]).to(torch.float32)
    Kg += (total * u)[None, :].to(torch.float32)
    return targets


def storage_dtype(w: Workload) -> torch.dtype:
    return torch.float32 if w.dtype == "f32" else torch.bfloat16


@dataclass
class Batch:
    """A whole layer: [B, H, rows, d] tensors in the storage dtype."""
    Q: torch.Tensor
    K: torch.Tensor
    V: torch.Tensor
    Kg: torch.Tensor
    Vg: torch.Tensor
    targets: list  # per unit (b*H + h): planted targets or None


def make_batch(w: Workload, layer: int = 0, planted: bool = True, device="cpu", cfg: str | None = None,
               units: list | None = None) -> Batch:
    """Draw every unit (or only `units`, others left zero) of one layer.  Q
    has heads * group query heads; query head h * group + g belongs to KV
    head h."""
    dt = storage_dtype(w)
    B, H, d, G = w.batch, w.heads, w.head_dim, w.group
    dev = torch.device(device)
    Q = torch.zeros(B, H * G, w.q, d, dtype=dt, device=dev)
    K = torch.zeros(B, H, w.n, d, dtype=dt, device=dev)
    V = torch.zeros(B, H, w.n, d, dtype=dt, device=dev)
    Kg = torch.zeros(B, H, w.ng, d, dtype=dt, device=dev)
    Vg = torch.zeros(B, H, w.ng, d, dtype=dt, device=dev)
    targets = [None] * (B * H)
    for b in range(B):
        for h in range(H):
            if units is not None and b * H + h not in units:
                continue
            u = make_unit(w, b, h, layer, planted, dev, cfg)
            Q[b, h * G:(h + 1) * G] = u.Q.to(dt).view(G, w.q, d)
            K[b, h] = u.K.to(dt)
            V[b, h] = u.V.to(dt)
            Kg[b, h] = u.Kg.to(dt)
            Vg[b, h] = u.Vg.to(dt)
            targets[b * H + h] = u.targets
    return Batch(Q, K, V, Kg, Vg, targets)


def make_batch_fast(w: Workload, layer: int = 0, device="cuda", seed_salt: int = 0) -> Batch:
    """Unplanted i.i.d. N(0,1) layer drawn in a few large calls (timing inputs
    for the 32-layer stack, where the per-unit generator would be slow)."""
    dt = storage_dtype(w)
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(unit_seed("c5", layer, 0, 0, 1 + seed_salt))
    B, H, d = w.batch, w.heads, w.head_dim

    def rn(rows, heads=H):
        return torch.randn(B, heads, rows, d, generator=g, device=dev, dtype=torch.float32).to(dt)

    return Batch(rn(w.q, w.q_heads), rn(w.n), rn(w.n), rn(w.ng), rn(w.ng), [None] * (B * H))
