"""Seeded synthetic KV streams shaped like the paper's workloads.

Only random numbers and shapes live here -- none of the eviction arithmetic --
so both the CUDA path and the fp64 oracle consume the same bytes.  The paper's
own inputs (RULER, LongBench, MATH-500 activations of real models) are not
available; these generators stand in for them with the head counts, head
dims, block sizes, budgets and context lengths of the paper's settings
(Sec. 4 protocol: B = 128 blocks plus per-step decode eviction; 2k/4k budgets;
65k LongBench contexts; 25% MATH-500 budgets; Table tab:gqa_ratios shapes).

Recipes (per (sequence, layer, KV head) unit u, per-coordinate N(0,1) noise z):

* ``gauss_outlier``  v = m_u + r z, m_u = N(0,1)^d * U[0.5, 2], r = exp(N(0, 0.5^2)),
  r *= 8 with probability 0.02 (outlier tokens).  K = m_k + a_u z' with
  a_u = sqrt(2) * sigma_V / ratio_u, sigma_V = 1.434 sqrt(d) (the std over
  tokens of |r z| for this r), so sigma_V / sigma_K ~= ratio_u.
* ``student_t``      v = m_u + |t_3| z (Student-t, nu = 3, one scale per token),
  sigma_V = 1.336 sqrt(d); K low-dispersion Gaussian with ratio 3.
* ``drift``          new tokens v_t = m_u(t) + z with a random-walk mean
  m_u(t+1) = m_u(t) + 0.02 N(0,1)^d; the initial cache uses ``gauss_outlier``.
* ``two_cluster``    centres c1, c2 = 2 N(0,1)^d per unit, v = c + 0.5 z with
  c = c1 (p = 0.8) or c2; strongly bimodal scores.  K Gaussian, ratio 2.

Tie stress (tests): ``dup_fraction`` copies that fraction of rows from
earlier rows of the same block (exact duplicates, hence exact score ties);
``small_int`` rounds values to integers in [-8, 8].
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

# The five workloads.  ``units`` = n_seq * n_layer * n_kv_head.
CONFIGS = {
    "tiny_prefill": dict(index=0, kind="prefill", gen="gauss_outlier", n_seq=1, n_layer=1,
                         n_kv_head=2, head_dim=64, T=512, B=32, N=128, ratio=(2.0, 2.0)),
    "prefill_gqa8b": dict(index=1, kind="prefill", gen="gauss_outlier", n_seq=1, n_layer=36,
                          n_kv_head=8, head_dim=128, T=32768, B=128, N=2048, ratio=(1.5, 4.0)),
    "prefill_wide": dict(index=2, kind="prefill", gen="student_t", n_seq=1, n_layer=42,
                         n_kv_head=8, head_dim=256, T=65536, B=256, N=4096, ratio=(3.0, 3.0)),
    "decode_batched": dict(index=3, kind="decode", gen="drift", n_seq=64, n_layer=32,
                           n_kv_head=8, head_dim=128, N=4096, steps=1024, check_every=64,
                           ratio=(1.5, 4.0)),
    "ratio_budget": dict(index=4, kind="ratio", gen="two_cluster", n_seq=16, n_layer=28,
                         n_kv_head=4, head_dim=128, prompt=512, B=128, gen_tokens=16384,
                         budget_ratio=0.25, ratio=(2.0, 2.0)),
}
BY_INDEX = {c["index"]: name for name, c in CONFIGS.items()}
BASE_SEED = 20260

SIGMA_V_PER_SQRT_D = {"gauss_outlier": 1.434, "student_t": 1.336, "drift": 1.434,
                      "two_cluster": 1.0}


def config(name_or_index):
    name = BY_INDEX[name_or_index] if isinstance(name_or_index, int) else name_or_index
    return name, dict(CONFIGS[name])


def units_of(cfg) -> int:
    return cfg["n_seq"] * cfg["n_layer"] * cfg["n_kv_head"]


def budget_at(cfg, total_tokens: int) -> int:
    """Ratio-budget rule: N_t = floor(ratio * L_t) tokens processed so far."""
    return max(1, int(math.floor(cfg["budget_ratio"] * total_tokens)))


@dataclass
class TokenStream:
    """Successive blocks of new K/V rows for ``units`` units.  Deterministic
    in (seed, sequence of calls); generated on ``device``."""

    gen: str
    units: int
    d: int
    device: str = "cuda"
    seed: int = BASE_SEED
    ratio: tuple = (2.0, 2.0)
    dup_fraction: float = 0.0
    small_int: bool = False
    _g: torch.Generator = field(init=False, repr=False)

    def __post_init__(self):
        self._g = torch.Generator(device=self.device)
        self._g.manual_seed(int(self.seed))
        U, d, dev, g = self.units, self.d, self.device, self._g
        scale = torch.rand(U, 1, generator=g, device=dev) * 1.5 + 0.5
        self.m = torch.randn(U, d, generator=g, device=dev) * scale
        self.m_k = torch.randn(U, d, generator=g, device=dev)
        lo, hi = self.ratio
        r = torch.rand(U, 1, generator=g, device=dev) * (hi - lo) + lo
        sigma_v = SIGMA_V_PER_SQRT_D[self.gen] * math.sqrt(d)
        self.a_k = math.sqrt(2.0) * sigma_v / r          # [U, 1] per-coordinate K noise scale
        if self.gen == "two_cluster":
            self.c1 = 2.0 * torch.randn(U, d, generator=g, device=dev)
            self.c2 = 2.0 * torch.randn(U, d, generator=g, device=dev)

    def _randn(self, *shape):
        return torch.randn(*shape, generator=self._g, device=self.device)

    def _values(self, B: int, initial: bool, units: slice) -> torch.Tensor:
        U = units.stop - units.start
        d = self.d
        z = self._randn(U, B, d)
        m = self.m[units].unsqueeze(1)
        kind = self.gen
        if kind == "drift" and initial:
            kind = "gauss_outlier"
        if kind == "gauss_outlier":
            r = torch.exp(0.5 * self._randn(U, B, 1))
            out = torch.rand(U, B, 1, generator=self._g, device=self.device) < 0.02
            r = torch.where(out, r * 8.0, r)
            return m + r * z
        if kind == "student_t":
            chi2 = (self._randn(U, B, 3) ** 2).sum(-1, keepdim=True)
            t = self._randn(U, B, 1) / torch.sqrt(chi2 / 3.0)
            return m + t.abs() * z
        if kind == "drift":
            # one random-walk step of the mean per new token
            steps = 0.02 * self._randn(U, B, d)
            walk = self.m[units].unsqueeze(1) + torch.cumsum(steps, dim=1)
            self.m[units] = walk[:, -1]
            return walk + z
        if kind == "two_cluster":
            pick = torch.rand(U, B, 1, generator=self._g, device=self.device) < 0.8
            c = torch.where(pick, self.c1[units].unsqueeze(1), self.c2[units].unsqueeze(1))
            return c + 0.5 * z
        raise ValueError(kind)

    def _finish(self, x: torch.Tensor) -> torch.Tensor:
        if self.small_int:
            x = torch.clamp(torch.round(x), -8, 8)
        if self.dup_fraction > 0 and x.shape[1] > 1:
            U, B, _ = x.shape
            dup = torch.rand(U, B, generator=self._g, device=self.device) < self.dup_fraction
            dup[:, 0] = False
            src = (torch.rand(U, B, generator=self._g, device=self.device)
                   * torch.arange(B, device=self.device)).long()
            gathered = torch.gather(x, 1, src.unsqueeze(-1).expand_as(x))
            x = torch.where(dup.unsqueeze(-1), gathered, x)
        return x.to(torch.bfloat16)

    def next(self, B: int, initial: bool = False, units: slice | None = None):
        """(k, v): bf16 [U, B, d] for the next B tokens of every unit (or of
        the unit range ``units``)."""
        units = units or slice(0, self.units)
        U = units.stop - units.start
        v = self._finish(self._values(B, initial, units))
        k = self.m_k[units].unsqueeze(1) + self.a_k[units].unsqueeze(1) * self._randn(U, B, self.d)
        return self._finish(k), v


def stream_for(cfg, device="cuda", seed=None, units=None, **kw) -> TokenStream:
    seed = BASE_SEED + cfg["index"] if seed is None else seed
    return TokenStream(gen=cfg["gen"], units=units or units_of(cfg), d=cfg["head_dim"],
                       device=device, seed=seed, ratio=cfg.get("ratio", (2.0, 2.0)), **kw)


def fill_rows(stream: TokenStream, k_units, v_units, n: int, chunk_units: int = 512,
              initial: bool = True) -> None:
    """Writes n fresh rows into slots [0, n) of [U, capacity, d] views, a few
    hundred units at a time (bounded temporaries for the large caches)."""
    U = k_units.shape[0]
    for u0 in range(0, U, chunk_units):
        sl = slice(u0, min(U, u0 + chunk_units))
        k, v = stream.next(n, initial=initial, units=sl)
        k_units[sl, :n].copy_(k)
        v_units[sl, :n].copy_(v)
