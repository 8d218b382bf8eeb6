"""Workload shapes of the compression step and their algorithmic byte / FLOP counts.

A workload names the model shape whose KV cache is compressed (layers, batch,
query / KV heads, head_dim), the cache length before and after one compress,
the recent window, the beacon count and the number of decode queries that reach
the beacons between two compresses.  The shapes follow the four models the
paper evaluates (Section 5.1): Qwen3-4B, R1-Distill-Llama-8B, Qwen3-14B and a
Qwen3-8B-shaped long decode trace; rope_theta is each model family's published
rotary base.

An *instance* is one (layer, batch row, KV head); all instances are
independent, so every count below is per instance times ``n_inst``.
"""
from __future__ import annotations

import dataclasses
import math


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    batch: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    L: int                    # cached tokens when the compress runs
    budget: int               # tokens kept
    window: int               # recent queries per query head == always-kept last tokens
    n_beacons: int            # beacons per KV head
    n_new: int                # decode queries per query head reaching the beacons before the compress
    n_init: int               # prompt queries per query head used for the FPS seed
    rope_theta: float
    n_clusters: int           # planted query clusters per instance
    sigma: float              # cluster spread (noise norm relative to the unit centre)
    noise_frac: float = 0.3   # share of isotropic (unclustered) queries
    k_offset_std: float = 0.0  # per-(layer, KV head) mean offset of the keys
    n_prefix: int = 0
    revisit_dirs: int = 0     # planted "revisit" directions per instance
    revisit_frac: float = 0.0  # share of new queries aimed at them
    revisit_keys: int = 0     # planted keys per direction, in the first 10% of the cache
    revisit_beta: float = 8.0
    # long decode trace (0 = single compress step)
    trace_steps: int = 0
    prefill: int = 0
    drift: float = 0.0

    # ----------------------------------------------------------- derived
    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def n_inst(self) -> int:
        return self.n_layers * self.batch * self.n_kv_heads

    @property
    def n_obs(self) -> int:
        """Scoring queries per instance: G * W recent + n_beacons beacons."""
        return self.group * self.window + self.n_beacons

    @property
    def capacity(self) -> int:
        return self.L

    def scaled(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    # ----------------------------------------------------------- accounting
    def compress_bytes(self) -> int:
        """Algorithmic HBM bytes of one compress over all instances.

        Read every cached key once (L*d*2), read the kept K and V rows and write
        them back (budget*d*2*4), read the recent queries (G*W*d*2) and write the
        kept indices (budget*4).  Evicted V rows are never read."""
        d = self.head_dim
        keep = min(self.budget, self.L)
        per = self.L * d * 2 + keep * d * 2 * 4 + self.group * self.window * d * 2 + keep * 4
        return per * self.n_inst

    def update_bytes(self, n_new: int | None = None) -> int:
        """Algorithmic HBM bytes of one beacon update: the new queries, the
        centroids read, and the touched centroids written (fp32)."""
        n_new = self.n_new if n_new is None else n_new
        d = self.head_dim
        nq = self.group * n_new
        per = nq * d * 2 + self.n_beacons * d * 4 + min(nq, self.n_beacons) * d * 4
        return per * self.n_inst

    def update_seq_bytes(self, n_steps: int) -> int:
        """Algorithmic HBM bytes of n_steps decode steps (one query per query head each) applied in one
        call: every step's queries, the centroids read once, the touched centroids written once."""
        d = self.head_dim
        nq = self.group * n_steps
        per = nq * d * 2 + self.n_beacons * d * 4 + min(nq, self.n_beacons) * d * 4
        return per * self.n_inst

    def compress_flops(self) -> int:
        return 2 * self.n_obs * self.L * self.head_dim * self.n_inst

    def update_flops(self, n_new: int | None = None) -> int:
        n_new = self.n_new if n_new is None else n_new
        return 2 * self.group * n_new * self.n_beacons * self.head_dim * self.n_inst

    def step_bytes(self) -> int:
        return self.compress_bytes() + self.update_bytes()

    def step_flops(self) -> int:
        return self.compress_flops() + self.update_flops()

    def tokens_per_step(self) -> int:
        """Cached KV tokens scored and compacted by one compress."""
        return self.n_inst * self.L

    def roofline_seconds(self, hbm_gbs: float, bf16_tflops: float) -> float:
        return max(self.step_bytes() / (hbm_gbs * 1e9), self.step_flops() / (bf16_tflops * 1e12))


TINY = Workload(
    name="tiny_1L_b1_h4kv2_d64_L1088_B512", n_layers=1, batch=1, n_q_heads=4, n_kv_heads=2, head_dim=64,
    L=1088, budget=512, window=8, n_beacons=4, n_new=64, n_init=64, rope_theta=1e4, n_clusters=4, sigma=0.1)

QWEN3_4B = Workload(
    name="qwen3_4b_36L_b16_L4224_B4096", n_layers=36, batch=16, n_q_heads=32, n_kv_heads=8, head_dim=128,
    L=4224, budget=4096, window=8, n_beacons=8, n_new=128, n_init=64, rope_theta=1e6, n_clusters=8, sigma=0.15,
    k_offset_std=0.5)

LLAMA_8B = Workload(
    name="r1_llama_8b_32L_b32_L2176_B2048", n_layers=32, batch=32, n_q_heads=32, n_kv_heads=8, head_dim=128,
    L=2176, budget=2048, window=8, n_beacons=16, n_new=128, n_init=64, rope_theta=5e5, n_clusters=16, sigma=0.15,
    k_offset_std=0.5)

QWEN3_14B = Workload(
    name="qwen3_14b_40L_b8_L8320_B8192", n_layers=40, batch=8, n_q_heads=40, n_kv_heads=8, head_dim=128,
    L=8320, budget=8192, window=8, n_beacons=16, n_new=128, n_init=64, rope_theta=1e6, n_clusters=16, sigma=0.15,
    k_offset_std=0.5, revisit_dirs=2, revisit_frac=0.05, revisit_keys=32)

QWEN3_8B_TRACE = Workload(
    name="qwen3_8b_trace_36L_b16_32768steps_B4096", n_layers=36, batch=16, n_q_heads=32, n_kv_heads=8,
    head_dim=128, L=4224, budget=4096, window=8, n_beacons=16, n_new=1, n_init=128, rope_theta=1e6,
    n_clusters=16, sigma=0.15, k_offset_std=0.5, trace_steps=32768, prefill=128, drift=0.005)

WORKLOADS = {1: TINY, 2: QWEN3_4B, 3: LLAMA_8B, 4: QWEN3_14B, 5: QWEN3_8B_TRACE}


def recent_positions(t_pos: int, window: int) -> list[int]:
    """Absolute positions of the W most recent decode queries ending at t_pos."""
    return [t_pos - window + 1 + w for w in range(window)]


def n_obs_padded(n_obs: int) -> int:
    """Scoring-query count rounded up to the tensor-core N granularity (16)."""
    return max(16, int(math.ceil(n_obs / 16.0)) * 16)
