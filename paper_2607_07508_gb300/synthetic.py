"""Seeded synthetic workloads for the SAO loss head.

This module only draws random inputs. It holds none of the loss head's
arithmetic (no logits, no softmax, no ratio, no GAE), so that the CUDA path
and the fp64 oracle can both consume the same draws without sharing any of
the method.

The workloads stand in for the paper's agentic trajectories (single rollout
per prompt, batch of packed variable-length trajectories up to 128k tokens,
§4.1 "Training Details"). Per-token and per-trajectory arrays are drawn with
numpy's PCG64 so they are identical on every machine. The two large dense
operands (hidden states ``H`` and LM-head weight ``W``) are drawn with a
seeded ``torch.Generator`` on the requested device; a parity comparison always
uses one generated copy for both sides.

Field meanings (row ``t`` of ``H`` predicts token ``y[t]``):

* ``cu_seqlens`` int32 [B+1]  packed trajectory offsets
* ``loss_mask``  uint8 [N]    1 = action token (model generated), 0 = prompt or
  observation token (environment output), §3.2 "Skip-Observation"
* ``values``     fp32 [N]     value-model outputs V(s_t)
* ``rewards``    fp32 [B]     terminal binary reward per trajectory
* ``y``          int32 [N]    sampled token ids, uniform over the vocabulary
* ``xi``         fp32 [N]     staleness of the rollout policy as a log-ratio:
  ``old_logp = logp + xi`` for whatever ``logp`` the caller holds, so the
  token ratio is ``exp(-xi)``
* ``logp_syn``   fp32 [N]     stand-in current-policy log-probs for exercising
  the policy loss on its own (not derived from H, W)
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Optional

import numpy as np

SEED_BASE = 2607_07508

# Hyper-parameters of the paper's runs (§4.1): clip bounds for reasoning and
# coding, the length-adaptive GAE factor and the critic's lambda.
PAPER_EPS_REASONING = (0.3, 5.0)
PAPER_EPS_CODING = (0.8, 3.0)
PAPER_ALPHA = 1.5
PAPER_LAMBDA_CRITIC = 1.0


@dataclasses.dataclass
class Workload:
    name: str
    N: int
    B: int
    h: int
    V: int
    dtype: str                      # "f32" or "bf16" for H, W
    cu_seqlens: np.ndarray
    loss_mask: np.ndarray
    values: np.ndarray
    rewards: np.ndarray
    y: np.ndarray
    xi: np.ndarray
    logp_syn: np.ndarray
    gamma: float
    lam: float
    lam_critic: float
    alpha: float
    eps_low: float
    eps_high: float
    H: object = None                 # torch tensor [N, h] or None
    W: object = None                 # torch tensor [V, h] or None
    recipe: str = ""

    @property
    def old_logp_syn(self) -> np.ndarray:
        return (self.logp_syn + self.xi).astype(np.float32)


# ---------------------------------------------------------------------------
# length and mask recipes
# ---------------------------------------------------------------------------

def _fit_total(lengths: np.ndarray, total: int, lo: int, hi: int) -> np.ndarray:
    """Rescale positive lengths so they sum to ``total`` exactly, each in [lo, hi]."""
    L = lengths.astype(np.float64)
    for _ in range(64):
        L = np.clip(L * (total / L.sum()), lo, hi)
        if abs(L.sum() - total) < 0.5:
            break
    L = np.floor(L).astype(np.int64)
    diff = total - int(L.sum())
    i = 0
    while diff != 0:
        j = i % len(L)
        if diff > 0 and L[j] < hi:
            L[j] += 1
            diff -= 1
        elif diff < 0 and L[j] > lo:
            L[j] -= 1
            diff += 1
        i += 1
        if i > 64 * len(L) + 4 * abs(diff) + 1024:
            raise ValueError("cannot fit lengths to total")
    return L


def lognormal_lengths(rng, total: int, median: int, max_len: int, min_len: int = 16,
                      sigma: float = 1.0) -> np.ndarray:
    draws = []
    acc = 0
    while acc < total:
        x = int(np.clip(rng.lognormal(math.log(median), sigma), min_len, max_len))
        draws.append(x)
        acc += x
    return _fit_total(np.array(draws), total, min_len, max_len)


def lognormal_lengths_n(rng, n: int, total: int, median: int, max_len: int, min_len: int = 16,
                        sigma: float = 1.0) -> np.ndarray:
    raw = np.clip(rng.lognormal(math.log(median), sigma, size=n), min_len, max_len)
    return _fit_total(raw, total, min_len, max_len)


def pareto_lengths(rng, n: int, total: int, lo: int, hi: int, shape: float = 1.5) -> np.ndarray:
    raw = lo * (1.0 + rng.pareto(shape, size=n))
    return _fit_total(np.clip(raw, lo, hi), total, lo, hi)


def turn_mask(rng, length: int, obs_frac: float, prompt_span: int = 0,
              mean_action: int = 256) -> np.ndarray:
    """Alternating action / observation turns: [prompt][a0][o0][a1][o1]...

    Action spans are geometric with mean ``mean_action``; observation spans are
    geometric with the mean that gives ``obs_frac`` of the non-prompt tokens.
    About one trajectory in four ends on an observation span.
    """
    m = np.zeros(length, np.uint8)
    pos = min(prompt_span, length)
    if obs_frac <= 0.0:
        m[pos:] = 1
        return m
    mean_obs = max(1.0, mean_action * obs_frac / max(1e-9, 1.0 - obs_frac))
    while pos < length:
        a = int(rng.geometric(1.0 / mean_action))
        m[pos:pos + a] = 1
        pos += a
        o = int(rng.geometric(1.0 / mean_obs))
        pos += o
    if rng.random() < 0.75:
        # most agentic traces end with the model's own final answer
        tail = min(length, int(rng.geometric(1.0 / mean_action)))
        m[length - tail:] = 1
    return m


def _pack(lengths: np.ndarray) -> np.ndarray:
    cu = np.zeros(len(lengths) + 1, np.int64)
    np.cumsum(lengths, out=cu[1:])
    return cu.astype(np.int32)


# ---------------------------------------------------------------------------
# dense operands
# ---------------------------------------------------------------------------

def dense_operands(N: int, V: int, h: int, dtype: str, seed: int, device="cpu",
                   w_std: float = 0.02):
    """H ~ N(0,1) [N,h] and W ~ N(0, w_std) [V,h], rounded to ``dtype``."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    H = torch.randn(N, h, generator=g, device=device, dtype=torch.float32).to(tdt)
    W = (torch.randn(V, h, generator=g, device=device, dtype=torch.float32) * w_std).to(tdt)
    return H, W


# ---------------------------------------------------------------------------
# the five workload configurations
# ---------------------------------------------------------------------------

CONFIG_NAMES = ("tiny", "small", "moe", "long", "large")


def _common_tail(rng, N, B, V, lengths, mask, val_mu, val_sd, p_reward):
    values = rng.normal(val_mu, val_sd, size=N).astype(np.float32)
    rewards = (rng.random(B) < p_reward).astype(np.float32)
    y = rng.integers(0, V, size=N, dtype=np.int64).astype(np.int32)
    logp_syn = (-rng.exponential(2.0, size=N)).astype(np.float32)
    return values, rewards, y, logp_syn


def make_workload(name: str, *, dense: bool = True, device="cpu", seed: Optional[int] = None,
                  N_override: Optional[int] = None) -> Workload:
    """Build one of the five configurations (tiny, small, moe, long, large).

    ``dense=False`` skips H and W (per-token arrays only). ``N_override``
    rescales the packed total (used for bandwidth studies of the O(N) kernels).
    """
    idx = CONFIG_NAMES.index(name)
    seed = SEED_BASE + idx if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(seed))

    if name == "tiny":
        h, V, dtype = 256, 4096, "f32"
        lengths = rng.integers(64, 513, size=8)
        N = int(lengths.sum())
        mask = np.ones(N, np.uint8)
        xi = rng.normal(0.0, 0.05, size=N)
        gamma, lam, lam_c, alpha, el, eh = 1.0, 1.0, 1.0, 0.0, 0.2, 0.28
        vm, vs, pr = 0.4, 0.2, 0.4
        recipe = "8 trajectories, uniform 64-512 tokens; xi~N(0,0.05); all action tokens"
    elif name == "small":
        h, V, dtype = 1024, 32000, "bf16"
        N = 98304 if N_override is None else N_override
        lengths = lognormal_lengths_n(rng, 64, N, 1024, 8192)
        mask = np.ones(N, np.uint8)
        stale = rng.random(N) < 0.3
        xi = np.where(stale, rng.normal(0.0, 0.1, size=N), 0.0)
        gamma, lam, lam_c, alpha, el, eh = 1.0, 1.0, 1.0, 0.0, 0.2, 0.28
        vm, vs, pr = 0.4, 0.2, 0.4
        recipe = "64 lognormal(median 1k, sigma 1) lengths clamp [16,8k] fit to 98304 tokens; xi~N(0,0.1) on 30%"
    elif name == "moe":
        h, V, dtype = 2048, 151936, "bf16"
        N = 65536 if N_override is None else N_override
        lengths = lognormal_lengths(rng, N, 4096, 32768)
        mask = np.concatenate([turn_mask(rng, int(L), 0.25) for L in lengths])
        k = rng.integers(1, 5, size=N)
        xi = rng.normal(0.0, 1.0, size=N) * 0.05 * k
        gamma, lam, lam_c, alpha = 1.0, 0.95, 1.0, 0.0
        el, eh = PAPER_EPS_REASONING
        vm, vs, pr = 0.4, 0.2, 0.4
        recipe = ("lognormal(median 4k, sigma 1) clamp [16,32k] to 65536 tokens; alternating "
                  "action/observation turns, 25% observation; xi~N(0,0.05k), k~U{1..4}")
    elif name == "long":
        h, V, dtype = 4096, 151936, "bf16"
        N = 524288 if N_override is None else N_override
        B0 = 16 if N_override is None else max(1, N // 32768)
        lo, hi = (16384, 131072) if N_override is None else (16, 131072)
        lengths = pareto_lengths(rng, B0, N, lo, hi)
        parts = []
        for L in lengths:
            prompt = int(min(L // 8, rng.integers(256, 2049)))
            parts.append(turn_mask(rng, int(L), 0.40, prompt_span=prompt))
        mask = np.concatenate(parts)
        xi = rng.normal(0.0, 0.05, size=N)
        gamma, lam, lam_c, alpha = 1.0, 1.0, PAPER_LAMBDA_CRITIC, PAPER_ALPHA
        el, eh = PAPER_EPS_CODING
        vm, vs, pr = 0.3, 0.25, 0.3
        recipe = ("16 Pareto(1.5)-tailed trajectories in [16k,128k] to 524288 tokens; masked prompt "
                  "span then alternating turns, 40% observation; length-adaptive lambda, alpha=1.5")
    elif name == "large":
        h, V, dtype = 6144, 154880, "bf16"
        N = 262144 if N_override is None else N_override
        lengths = lognormal_lengths_n(rng, 128, N, 2048, 65536)
        mask = np.ones(N, np.uint8)
        el, eh = PAPER_EPS_REASONING
        xi = rng.normal(0.0, 0.05, size=N)
        push = rng.random(N) < 0.10
        low = rng.random(N) < 0.5
        r_lo = rng.uniform(0.3, 0.6, size=N) * (1.0 - el)
        r_hi = (1.0 + eh) * rng.uniform(1.1, 1.5, size=N)
        r_target = np.where(low, r_lo, r_hi)
        xi = np.where(push, -np.log(r_target), xi)
        gamma, lam, lam_c, alpha = 1.0, 1.0, 1.0, 0.0
        vm, vs, pr = 0.4, 0.2, 0.4
        recipe = ("128 lognormal(median 2k, sigma 1) lengths clamp [16,64k] fit to 262144 tokens; 10% of tokens "
                  "with a target ratio outside the clip bounds, the rest xi~N(0,0.05)")
    else:
        raise KeyError(name)

    lengths = np.asarray(lengths, np.int64)
    B = len(lengths)
    N = int(lengths.sum())
    cu = _pack(lengths)
    values, rewards, y, logp_syn = _common_tail(rng, N, B, V, lengths, mask, vm, vs, pr)
    wl = Workload(name=name, N=N, B=B, h=h, V=V, dtype=dtype, cu_seqlens=cu,
                  loss_mask=mask.astype(np.uint8), values=values, rewards=rewards, y=y,
                  xi=np.asarray(xi, np.float32), logp_syn=logp_syn, gamma=gamma, lam=lam,
                  lam_critic=lam_c, alpha=alpha, eps_low=el, eps_high=eh, recipe=recipe)
    if dense:
        wl.H, wl.W = dense_operands(N, V, h, dtype, seed + 1000, device=device)
    return wl


def make_custom(N_lengths, h: int, V: int, dtype: str, seed: int, *, obs_frac: float = 0.25,
                dense: bool = True, device="cpu", eps=(0.2, 0.28), gamma=1.0, lam=0.95,
                lam_critic=1.0, alpha=0.0, xi_sd=0.05) -> Workload:
    """A small workload with explicit trajectory lengths (ragged tails, empty trajectories)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    lengths = np.asarray(N_lengths, np.int64)
    B = len(lengths)
    N = int(lengths.sum())
    mask = np.concatenate([turn_mask(rng, int(L), obs_frac, mean_action=16) if L > 0
                           else np.zeros(0, np.uint8) for L in lengths]) if B else np.zeros(0, np.uint8)
    xi = rng.normal(0.0, xi_sd, size=N).astype(np.float32)
    values, rewards, y, logp_syn = _common_tail(rng, N, B, V, lengths, mask, 0.4, 0.2, 0.4)
    wl = Workload(name=f"custom{seed}", N=N, B=B, h=h, V=V, dtype=dtype, cu_seqlens=_pack(lengths),
                  loss_mask=mask.astype(np.uint8), values=values, rewards=rewards, y=y, xi=xi,
                  logp_syn=logp_syn, gamma=gamma, lam=lam, lam_critic=lam_critic, alpha=alpha,
                  eps_low=eps[0], eps_high=eps[1], recipe="explicit lengths")
    if dense and N > 0:
        wl.H, wl.W = dense_operands(N, V, h, dtype, seed + 1000, device=device)
    return wl


def bandwidth_workload(N: int = 1 << 27, B: int = 1 << 14, seed: int = SEED_BASE + 99) -> Workload:
    """Per-token arrays only, for the HBM study of the O(N) kernels: N tokens in B
    trajectories (lognormal lengths), moe-like masks, staleness and clip bounds."""
    rng = np.random.Generator(np.random.PCG64(seed))
    med = max(16, N // B // 2)
    lengths = lognormal_lengths(rng, N, med, max(64, 16 * med))
    B = len(lengths)
    # alternating action / observation turns as in the five configurations
    # (geometric spans, action mean 256 tokens, observation mean 128: one
    # third observation tokens), drawn vectorised over the whole batch
    n_turns = 2 * (N // 384 + 64)
    spans = np.empty(n_turns, np.int64)
    spans[0::2] = rng.geometric(1.0 / 256.0, size=n_turns // 2)
    spans[1::2] = rng.geometric(1.0 / 128.0, size=n_turns // 2)
    while spans.sum() < N:
        spans = np.concatenate([spans, spans])
    kind = np.tile(np.array([1, 0], np.uint8), len(spans) // 2)
    mask = np.repeat(kind, spans)[:N]
    values = rng.standard_normal(N, dtype=np.float32) * np.float32(0.2) + np.float32(0.4)
    rewards = (rng.random(B) < 0.4).astype(np.float32)
    xi = rng.standard_normal(N, dtype=np.float32) * np.float32(0.1)
    logp_syn = (-rng.standard_exponential(N, dtype=np.float32) * np.float32(2.0))
    return Workload(name="bandwidth", N=N, B=B, h=0, V=0, dtype="bf16", cu_seqlens=_pack(lengths),
                    loss_mask=mask, values=values, rewards=rewards,
                    y=np.zeros(0, np.int32), xi=xi, logp_syn=logp_syn, gamma=1.0, lam=0.95,
                    lam_critic=1.0, alpha=0.0, eps_low=PAPER_EPS_REASONING[0],
                    eps_high=PAPER_EPS_REASONING[1],
                    recipe=f"{N} tokens, {B} lognormal trajectories, alternating turns")


def describe(wl: Workload) -> Dict[str, object]:
    return {"workload": wl.name, "tokens": wl.N, "trajectories": wl.B, "hidden": wl.h,
            "vocab": wl.V, "dtype": wl.dtype, "eps_low": wl.eps_low, "eps_high": wl.eps_high,
            "gamma": wl.gamma, "lambda": wl.lam, "lambda_critic": wl.lam_critic,
            "alpha": wl.alpha}
