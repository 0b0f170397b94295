"""Seeded synthetic inputs for one ReTrace round (shared by tests and bench).

This module only draws random numbers and plants a known accepted prefix; it
holds none of the round's arithmetic (no argmax, no projection, no gate).  It
stands in for the paper's Qwen3-4B / Qwen3-8B + DFlash-b16 workloads on its
seven benchmarks (Sec. 5 "Models and Benchmarks"; Appendix "Model and ReTrace
Configuration"), whose weights and prompts are not available here: shapes,
value distributions and acceptance patterns follow those workloads.

Recipe for every tensor (seed 42, the paper's seed, plus a per-config offset):

* ``draft``  int32 [B, K], uniform over [0, V).
* ``logits`` [B, K+1, V], N(0, std^2) rounded to the storage dtype.  A design
  prefix length ``a_b`` is drawn per sequence (Uniform{0..K}, or Geometric(p)
  on {0, 1, ...} capped at K).  Rows i < a_b get logits[b, i, draft] = row
  max + 1, so the draft token is the unique row maximum; row a_b (if a_b < K)
  gets logits[b, a_b, draft] = row min - 1, so the draft token cannot win.
  With ``ties``: accepted rows also receive a copy of the maximum at a higher
  index (draft + delta) and the mismatch row receives the new maximum at the
  draft token AND at a lower index (draft - delta), with deltas inside one
  16-byte vector, across vectors and far apart.  The planted ``a_b`` is a
  design value; the oracle's accepted length is the truth.
* ``hD``, ``hT`` [B, K, d] N(0, 1); ``e`` one mask embedding [d] N(0, 0.02^2)
  broadcast over positions (DFlash proposal inputs are mask embeddings).
* ``Wc`` [d, 2d], ``Wv`` [d, d], ``Wg`` [d, 2d]: Xavier-uniform
  U(-a, a), a = sqrt(6 / (fan_in + fan_out)); ``beta`` = 1 (inference value).
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import torch

SEED = 42


@dataclass(frozen=True)
class RoundConfig:
    """Shape and distribution of one synthetic round workload."""

    name: str
    B: int
    K: int
    V: int
    d: int
    dtype: str  # "f32" or "bf16"
    logits_std: float
    prefix: str  # "uniform" or "geometric"
    prefix_p: float = 0.0
    ties: bool = False
    seed_offset: int = 0

    @property
    def torch_dtype(self) -> torch.dtype:
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def logits_bytes(self) -> int:
        return self.B * (self.K + 1) * self.V * self.elem_bytes


# The five workloads: a tiny fp32 case, then Qwen3-4B (d 2560) and Qwen3-8B
# (d 4096) shapes with the Qwen3 vocabulary (151936) and DFlash-b16 blocks.
CONFIGS = {
    1: RoundConfig("tiny-f32-B1-K8-V1024-d256", 1, 8, 1024, 256, "f32", 1.0, "uniform", seed_offset=1),
    2: RoundConfig("qwen3-4b-B1-K16", 1, 16, 151936, 2560, "bf16", 1.0, "geometric", 0.3, seed_offset=2),
    3: RoundConfig("qwen3-8b-B8-K16", 8, 16, 151936, 4096, "bf16", 2.0, "geometric", 0.3, seed_offset=3),
    4: RoundConfig("qwen3-4b-B64-K16-ties", 64, 16, 151936, 2560, "bf16", 1.0, "uniform", ties=True, seed_offset=4),
    5: RoundConfig("qwen3-8b-B256-K16", 256, 16, 151936, 4096, "bf16", 1.0, "geometric", 0.2, seed_offset=5),
}

# A half-size serving batch with config 5's per-sequence distributions, for
# multi-pass profiler captures (inputs still larger than L2, under 1 GB held).
PROFILE_CONFIG = RoundConfig("profile-qwen3-8b-B128-K16", 128, 16, 151936, 4096, "bf16", 1.0, "geometric", 0.2,
                             seed_offset=6)

# Offsets (in elements) at which copies of the row maximum are planted when
# ``ties`` is set: same 16-byte vector, next vector, a few KB away, far away.
TIE_DELTAS = (1, 3, 7, 8, 9, 61, 1024, 4093, 65537)


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _uniform(shape, g, device, lo=0.0, hi=1.0):
    return torch.rand(shape, generator=g, device=device, dtype=torch.float32) * (hi - lo) + lo


def draw_prefix(cfg: RoundConfig, g: torch.Generator, device) -> torch.Tensor:
    """Design accepted-prefix length per sequence (int64 [B], values 0..K)."""
    if cfg.prefix == "uniform":
        return torch.randint(0, cfg.K + 1, (cfg.B,), generator=g, device=device)
    # Geometric(p) on {0, 1, ...}: P(a >= k) = (1-p)^k, by inversion, capped at K.
    u = _uniform((cfg.B,), g, device).double().clamp_min(1e-300)
    a = torch.floor(torch.log(u) / math.log1p(-cfg.prefix_p))
    return a.clamp(max=cfg.K).long()


def make_round_inputs(cfg: RoundConfig, device="cpu", seed: int | None = None) -> dict:
    """Seeded tensors for one round of ``cfg`` on ``device``."""
    seed = SEED + 1000 * cfg.seed_offset if seed is None else seed
    g = _gen(device, seed)
    B, K, V, d = cfg.B, cfg.K, cfg.V, cfg.d
    dt = cfg.torch_dtype

    draft = torch.randint(0, V, (B, K), generator=g, device=device, dtype=torch.int64)
    a = draw_prefix(cfg, g, device)

    logits = torch.empty((B, K + 1, V), dtype=dt, device=device)
    for b in range(B):  # one sequence at a time bounds the fp32 temporary
        logits[b] = (torch.randn((K + 1, V), generator=g, device=device) * cfg.logits_std).to(dt)
    plant_prefix(logits, draft, a, ties=cfg.ties)

    hD = torch.randn((B, K, d), generator=g, device=device).to(dt)
    hT = torch.randn((B, K, d), generator=g, device=device).to(dt)
    e = (torch.randn((d,), generator=g, device=device) * 0.02).to(dt)
    Wc = xavier_uniform((d, 2 * d), g, device).to(dt)
    Wv = xavier_uniform((d, d), g, device).to(dt)
    Wg = xavier_uniform((d, 2 * d), g, device).to(dt)
    return {
        "cfg": cfg,
        "logits": logits,
        "draft": draft.to(torch.int32),
        "planted_prefix": a,
        "hD": hD,
        "hT": hT,
        "e": e,
        "Wc": Wc,
        "Wv": Wv,
        "Wg": Wg,
        "beta": 1.0,
    }


LOWRANK_LATENT = 64  # ranks of the low-rank conditioning weights (Appendix "Concurrent-Serving Experiment")
LOWRANK_CORRECTION = 32


def make_lowrank_weights(cfg: RoundConfig, device="cpu", seed: int | None = None) -> dict:
    """Seeded Xavier-uniform weights of the low-rank conditioning path for ``cfg``:
    P [64, d], B_c [32, 64 + d], A_c [64, 32], W_v [d, 64], W_g [d, d + 64]."""
    seed = SEED + 1000 * cfg.seed_offset + 7 if seed is None else seed
    g = _gen(device, seed)
    d, Lr, Cr, dt = cfg.d, LOWRANK_LATENT, LOWRANK_CORRECTION, cfg.torch_dtype
    return {
        "P": xavier_uniform((Lr, d), g, device).to(dt),
        "Bc": xavier_uniform((Cr, Lr + d), g, device).to(dt),
        "Ac": xavier_uniform((Lr, Cr), g, device).to(dt),
        "Wv_lr": xavier_uniform((d, Lr), g, device).to(dt),
        "Wg_lr": xavier_uniform((d, d + Lr), g, device).to(dt),
    }


SAMPLING = {"temperature": 1.0, "top_k": 20, "top_p": 0.95}  # Appendix "Evaluation Protocol", temperature 1


def make_sampled_inputs(cfg: RoundConfig, target_logits: torch.Tensor, device="cpu", seed: int | None = None,
                        draft_noise: float = 0.7) -> dict:
    """Drafter logits, draft tokens and uniforms for sampled verification of
    ``target_logits`` [B, K+1, V]: the drafter's logits are the target's plus
    N(0, (draft_noise * std)^2) noise, each draft token is one of its row's
    eight largest drafter logits (uniformly), and the uniforms are U[0, 1)."""
    seed = SEED + 1000 * cfg.seed_offset + 11 if seed is None else seed
    g = _gen(device, seed)
    B, K, V = cfg.B, cfg.K, cfg.V
    dl = torch.empty((B, K, V), dtype=target_logits.dtype, device=device)
    draft = torch.empty((B, K), dtype=torch.int32, device=device)
    for b in range(B):  # one sequence at a time bounds the fp32 temporary
        noise = torch.randn((K, V), generator=g, device=device) * (draft_noise * cfg.logits_std)
        row = target_logits[b, :K].float() + noise
        dl[b] = row.to(target_logits.dtype)
        top8 = torch.topk(dl[b].float(), 8, dim=-1).indices
        pick = torch.randint(0, 8, (K, 1), generator=g, device=device)
        draft[b] = torch.gather(top8, 1, pick)[:, 0].to(torch.int32)
    uniforms = torch.rand((B, K + 1), generator=g, device=device, dtype=torch.float32)
    return {"draft_logits": dl, "draft": draft, "uniforms": uniforms, **SAMPLING}


def xavier_uniform(shape, g, device) -> torch.Tensor:
    """U(-a, a) with a = sqrt(6 / (fan_in + fan_out)) for a [fan_out, fan_in] matrix."""
    fan_out, fan_in = shape
    bound = math.sqrt(6.0 / (fan_in + fan_out))
    return _uniform(shape, g, device, -bound, bound)


def plant_prefix(logits: torch.Tensor, draft: torch.Tensor, a: torch.Tensor, ties: bool = False) -> None:
    """Make the draft token the unique maximum of rows i < a_b and a loser of row a_b.

    With ``ties``, additionally plant equal maxima: at higher indices in the
    accepted rows (the draft token must still win: lowest index) and at a
    lower index in the mismatch row (that lower index must win).
    """
    B, K1, V = logits.shape
    K = K1 - 1
    dev = logits.device
    draft = draft.to(dev).long()
    a = a.to(dev).long()
    rowmax = logits.amax(dim=-1).float()  # [B, K+1]; max is exact in any dtype
    rowmin = logits.amin(dim=-1).float()
    slot = torch.arange(K, device=dev)[None, :].expand(B, K)
    bidx = torch.arange(B, device=dev)[:, None].expand(B, K)
    acc = slot < a[:, None]  # accepted rows
    bi, ii, tok = bidx[acc], slot[acc], draft[:, :K][acc]
    logits[bi, ii, tok] = (rowmax[bi, ii] + 1.0).to(logits.dtype)
    if ties:
        for k, delta in enumerate(TIE_DELTAS):
            sel = ((ii + k) % 3 == 0) & (tok + delta < V)
            logits[bi[sel], ii[sel], tok[sel] + delta] = logits[bi[sel], ii[sel], tok[sel]]
    mis = a < K  # sequences with a mismatch row a_b
    mb = torch.nonzero(mis).flatten()
    if mb.numel() == 0:
        return
    ma = a[mb]
    mtok = draft[mb, ma.clamp(max=K - 1)]
    if ties:
        deltas = torch.tensor(TIE_DELTAS, device=dev)[(mb + ma) % len(TIE_DELTAS)]
        lower_ok = mtok > 0
        top = (rowmax[mb, ma] + 1.0).to(logits.dtype)
        lb, la, lt = mb[lower_ok], ma[lower_ok], mtok[lower_ok]
        lower = (lt - deltas[lower_ok]).clamp(min=0)
        logits[lb, la, lt] = top[lower_ok]
        logits[lb, la, lower] = top[lower_ok]
        rest = ~lower_ok
        mb, ma, mtok = mb[rest], ma[rest], mtok[rest]
    if V > 1 and mb.numel() > 0:
        logits[mb, ma, mtok] = (rowmin[mb, ma] - 1.0).to(logits.dtype)


def as_bits_numpy(t: torch.Tensor):
    """Host copy of a tensor as numpy: bf16 as uint16 bit patterns, others as-is."""
    t = t.detach().to("cpu").contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view("uint16")
    return t.numpy()
