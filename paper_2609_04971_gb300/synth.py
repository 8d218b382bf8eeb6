"""Seeded synthetic inputs shaped like the paper's reasoning-model decode traces.

This module only draws random numbers and lays them out; it holds none of the
compression step's arithmetic, and both the CUDA path and the CPU oracle
consume what it produces.  Everything is seeded per tensor, so a workload is
reproducible on any device (the stream of numbers differs between CPU and
CUDA generators; tests copy device inputs to the host for the oracle).

Recipe (the stand-in for AIME24 / MATH-500 / LiveCodeBench / GPQA-Diamond
traces, which are not available):
  * keys:    bf16(N(0, 1) + mu), mu ~ N(0, k_offset_std^2 I_d) per (layer, KV head);
  * values:  bf16(N(0, 1));
  * queries (pre-RoPE): per instance, n_clusters unit centres c_k; a query is
    isotropic noise rho * xi / sqrt(d) with probability noise_frac, otherwise
    rho * (c_k + sigma * xi / sqrt(d)) for a uniform k; rho = sqrt(d) so that
    logits have about unit spread.  Global queries clustering in pre-RoPE
    space is the observation of Section 3.2;
  * revisit workloads additionally plant directions u_r supported on the 16
    lowest-frequency rotary pairs (where rotation at any position of these
    workloads turns a vector by < 0.3 rad, so no rotation is needed to keep
    them aligned), aim revisit_frac of the new queries at them and plant
    revisit_keys keys beta * u_r + 0.1 xi per direction in the first 10% of
    the cache;
  * trace workloads drift every centre by c <- normalise(c + drift * xi / sqrt(d))
    per decode step.
Layouts: queries [layers, batch, q_heads, n, d]; K and V [layers, batch,
kv_heads, capacity, d]; all bf16.
"""
from __future__ import annotations

import math
import zlib

import torch

from .workloads import Workload


def _generator(seed: int, wl: Workload, tag: str, device) -> torch.Generator:
    key = zlib.crc32(f"{seed}/{wl.name}/{tag}".encode())
    g = torch.Generator(device=device)
    g.manual_seed(key)
    return g


def _unit(x: torch.Tensor) -> torch.Tensor:
    return x / x.norm(dim=-1, keepdim=True).clamp_min(1e-30)


def cluster_centres(wl: Workload, seed: int, device) -> torch.Tensor:
    """Unit centres [layers, batch, kv_heads, n_clusters, d] (fp32)."""
    g = _generator(seed, wl, "centres", device)
    c = torch.randn(wl.n_layers, wl.batch, wl.n_kv_heads, wl.n_clusters, wl.head_dim, generator=g,
                    device=device, dtype=torch.float32)
    return _unit(c)


def revisit_directions(wl: Workload, seed: int, device) -> torch.Tensor | None:
    """Unit directions [layers, batch, kv_heads, revisit_dirs, d] on the low-frequency rotary pairs."""
    if wl.revisit_dirs == 0:
        return None
    g = _generator(seed, wl, "revisit_dirs", device)
    d, h = wl.head_dim, wl.head_dim // 2
    n_low = min(16, h)
    u = torch.zeros(wl.n_layers, wl.batch, wl.n_kv_heads, wl.revisit_dirs, d, device=device)
    z = torch.randn(wl.n_layers, wl.batch, wl.n_kv_heads, wl.revisit_dirs, 2 * n_low, generator=g, device=device)
    u[..., h - n_low:h] = z[..., :n_low]
    u[..., d - n_low:d] = z[..., n_low:]
    return _unit(u)


def _queries_from(centres: torch.Tensor, wl: Workload, n: int, g: torch.Generator,
                  revisit: torch.Tensor | None = None, revisit_frac: float = 0.0) -> torch.Tensor:
    """Mixture queries for one layer slice of centres [B, Hkv, C, d] -> bf16 [B, Hq, n, d]."""
    B, Hkv, C, d = centres.shape
    G = wl.group
    dev = centres.device
    rho = math.sqrt(d)
    cen = centres.repeat_interleave(G, dim=1)                       # [B, Hq, C, d]
    k = torch.randint(0, C, (B, Hkv * G, n), generator=g, device=dev)
    pick = torch.gather(cen, 2, k.unsqueeze(-1).expand(B, Hkv * G, n, d))
    xi = torch.randn(B, Hkv * G, n, d, generator=g, device=dev)
    u = torch.rand(B, Hkv * G, n, generator=g, device=dev)
    clustered = rho * (pick + wl.sigma * xi / math.sqrt(d))
    noise = rho * xi / math.sqrt(d)
    q = torch.where((u < wl.noise_frac).unsqueeze(-1), noise, clustered)
    if revisit is not None and revisit_frac > 0.0:
        R = revisit.shape[2]
        rv = revisit.repeat_interleave(G, dim=1)                    # [B, Hq, R, d]
        r = torch.randint(0, R, (B, Hkv * G, n), generator=g, device=dev)
        rpick = torch.gather(rv, 2, r.unsqueeze(-1).expand(B, Hkv * G, n, d))
        xr = torch.randn(B, Hkv * G, n, d, generator=g, device=dev)
        ur = torch.rand(B, Hkv * G, n, generator=g, device=dev)
        q = torch.where((ur < revisit_frac).unsqueeze(-1), rho * (rpick + wl.sigma * xr / math.sqrt(d)), q)
    return q.to(torch.bfloat16)


def queries(wl: Workload, seed: int, tag: str, n: int, device, centres: torch.Tensor | None = None,
            with_revisit: bool = False) -> torch.Tensor:
    """Pre-RoPE queries bf16 [layers, batch, q_heads, n, d] drawn per the recipe."""
    if centres is None:
        centres = cluster_centres(wl, seed, device)
    rv = revisit_directions(wl, seed, device) if with_revisit else None
    g = _generator(seed, wl, tag, device)
    out = torch.empty(wl.n_layers, wl.batch, wl.n_q_heads, n, wl.head_dim, dtype=torch.bfloat16, device=device)
    for l in range(wl.n_layers):
        out[l] = _queries_from(centres[l], wl, n, g, None if rv is None else rv[l],
                               wl.revisit_frac if with_revisit else 0.0)
    return out


def keys_values(wl: Workload, seed: int, device, capacity: int | None = None, rows: int | None = None):
    """K and V bf16 [layers, batch, kv_heads, capacity, d]; rows beyond ``rows`` are zero.

    Returns (K, V, planted) where planted is None or an int64 tensor
    [layers, batch, kv_heads, revisit_dirs * revisit_keys] of planted key positions."""
    cap = wl.capacity if capacity is None else capacity
    rows = cap if rows is None else rows
    d = wl.head_dim
    gk = _generator(seed, wl, "K", device)
    gv = _generator(seed, wl, "V", device)
    gm = _generator(seed, wl, "K_offset", device)
    K = torch.zeros(wl.n_layers, wl.batch, wl.n_kv_heads, cap, d, dtype=torch.bfloat16, device=device)
    V = torch.zeros_like(K)
    mu = wl.k_offset_std * torch.randn(wl.n_layers, 1, wl.n_kv_heads, 1, d, generator=gm, device=device)
    for l in range(wl.n_layers):
        K[l, :, :, :rows] = (torch.randn(wl.batch, wl.n_kv_heads, rows, d, generator=gk, device=device)
                             + mu[l]).to(torch.bfloat16)
        V[l, :, :, :rows] = torch.randn(wl.batch, wl.n_kv_heads, rows, d, generator=gv,
                                        device=device).to(torch.bfloat16)
    planted = None
    if wl.revisit_dirs > 0 and wl.revisit_keys > 0:
        rv = revisit_directions(wl, seed, device)
        gp = _generator(seed, wl, "planted", device)
        span = max(wl.revisit_dirs * wl.revisit_keys, rows // 10)
        n_pl = wl.revisit_dirs * wl.revisit_keys
        planted = torch.empty(wl.n_layers, wl.batch, wl.n_kv_heads, n_pl, dtype=torch.int64, device=device)
        for l in range(wl.n_layers):
            scores = torch.rand(wl.batch, wl.n_kv_heads, span, generator=gp, device=device)
            pos = scores.argsort(dim=-1)[..., :n_pl]                      # distinct positions
            direction = rv[l].repeat_interleave(wl.revisit_keys, dim=2)   # [B, Hkv, n_pl, d]
            kk = wl.revisit_beta * direction + 0.1 * torch.randn(
                wl.batch, wl.n_kv_heads, n_pl, d, generator=gp, device=device)
            K[l].scatter_(2, pos.unsqueeze(-1).expand(-1, -1, -1, d), kk.to(torch.bfloat16))
            planted[l] = pos
    return K, V, planted


def step_inputs(wl: Workload, seed: int = 0, device="cpu") -> dict:
    """Everything one update + compress step consumes, for a single-step workload.

    Keys: q_init, q_new, q_recent (bf16 queries), K, V (bf16 cache), planted,
    t_pos (absolute position of the newest token = L - 1) and recent_pos."""
    centres = cluster_centres(wl, seed, device)
    K, V, planted = keys_values(wl, seed, device)
    t_pos = wl.L - 1
    return dict(
        q_init=queries(wl, seed, "q_init", wl.n_init, device, centres),
        q_new=queries(wl, seed, "q_new", wl.n_new, device, centres, with_revisit=wl.revisit_dirs > 0),
        q_recent=queries(wl, seed, "q_recent", wl.window, device, centres),
        K=K, V=V, planted=planted, t_pos=t_pos,
        recent_pos=[t_pos - wl.window + 1 + w for w in range(wl.window)],
    )


class TraceGen:
    """Per-step inputs of a long decode trace (drifting clusters, one token per step)."""

    def __init__(self, wl: Workload, seed: int = 0, device="cpu"):
        self.wl = wl
        self.device = device
        self.centres = cluster_centres(wl, seed, device)
        self.g_q = _generator(seed, wl, "trace_q", device)
        self.g_kv = _generator(seed, wl, "trace_kv", device)
        self.g_drift = _generator(seed, wl, "trace_drift", device)
        gm = _generator(seed, wl, "K_offset", device)
        self.mu = wl.k_offset_std * torch.randn(wl.n_layers, 1, wl.n_kv_heads, 1, wl.head_dim, generator=gm,
                                                device=device)
        self.seed = seed

    def prefill(self):
        """(q_init [.., n_init, d], K rows [.., prefill, d], V rows) for the prompt."""
        wl = self.wl
        q_init = queries(wl, self.seed, "trace_q_init", wl.n_init, self.device, self.centres)
        k, v = self.kv_rows(wl.prefill)
        return q_init, k, v

    def kv_rows(self, n: int):
        wl = self.wl
        shape = (wl.n_layers, wl.batch, wl.n_kv_heads, n, wl.head_dim)
        k = (torch.randn(*shape, generator=self.g_kv, device=self.device) + self.mu).to(torch.bfloat16)
        v = torch.randn(*shape, generator=self.g_kv, device=self.device).to(torch.bfloat16)
        return k, v

    def step_queries(self) -> torch.Tensor:
        """One decode query per query head [layers, batch, q_heads, 1, d]; then the centres drift."""
        wl = self.wl
        q = torch.empty(wl.n_layers, wl.batch, wl.n_q_heads, 1, wl.head_dim, dtype=torch.bfloat16,
                        device=self.device)
        for l in range(wl.n_layers):
            q[l] = _queries_from(self.centres[l], wl, 1, self.g_q)
        if wl.drift > 0.0:
            xi = torch.randn(self.centres.shape, generator=self.g_drift, device=self.device)
            self.centres = _unit(self.centres + wl.drift * xi / math.sqrt(wl.head_dim))
        return q


def to_bits(t: torch.Tensor):
    """bf16 tensor -> numpy uint16 bit patterns (host copy)."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view("uint16")
