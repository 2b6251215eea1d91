"""Seeded synthetic inputs shaped like the paper's agentic RL batches.

This module feeds both the CUDA library and the float64 oracle; it holds none
of the method's arithmetic (no ratio, mask, clip, loss, gradient or EWMA
step).  It draws policy logits, perturbs them into "old" logits, samples the
rollout tokens from the old policy (Gumbel-max), and emulates the inference
engine's log-probabilities mu_old as the old policy's log-softmax at the
sampled token plus noise (torch.log_softmax places mu_old near pi_old; both
sides then receive mu_old as an input).  Sequence structure (lengths, prompt
masks, group-normalised advantages) follows the GRPO-style setting of the
paper's experiments (Sec. 6.1); the datasets and models themselves are not
used, and the vocabulary size V = 151936 matches the Qwen3 backbones.

Workloads (names say what they are):
  tiny_f32_v4096      T=256 (4 x 64), V=4096, fp32; logits N(0,2^2), old = +N(0,0.1^2),
                      mu noise N(0,0.05^2), advantages from Bernoulli(0.5) rewards,
                      groups of 4; band [0.5, 2], eps 0.2 / 0.28
  grpo_bf16_v32000    T=65536 (64 x 1024), V=32000, bf16; logits N(0,3^2) + 8 at one
                      random id per row, old = +N(0,0.2^2), mu noise N(0,0.02^2),
                      Bernoulli(0.3) rewards in groups of 8; band [0.5, 2]
  agentic_bf16_v151936  T=65536 packed from 128 sequences of length U[64,1024]
                      (prompt prefix U[0, L/4] and padding masked out), V=151936,
                      bf16, distributions as grpo; groups of 8 sequences; band [0.8, 1.25]
  heavytail_bf16_v151936  T=16384, V=151936, bf16; as grpo but 10% of rows peak +20,
                      mu noise 0.1 * Student-t(2), advantages N(0,1) per token; band [0.5, 2]
  EWMA buffers        n fp32 parameters theta ~ N(0, 0.02^2), theta_prox = theta + N(0, 1e-4^2)
"""

from dataclasses import dataclass, field

import numpy as np
import torch

V_QWEN3 = 151936
EWMA_N_7B = 7_600_000_000

WORKLOADS = {
    "tiny_f32_v4096": dict(
        T=256, V=4096, dtype=torch.float32, z_std=2.0, peak=0.0, heavy_frac=0.0, heavy_peak=0.0,
        old_std=0.1, mu=("normal", 0.05), adv=("grpo", 0.5, 4), layout=("fixed", 64),
        band=(0.5, 2.0), eps=(0.2, 0.28)),
    "grpo_bf16_v32000": dict(
        T=65536, V=32000, dtype=torch.bfloat16, z_std=3.0, peak=8.0, heavy_frac=0.0,
        heavy_peak=0.0, old_std=0.2, mu=("normal", 0.02), adv=("grpo", 0.3, 8),
        layout=("fixed", 1024), band=(0.5, 2.0), eps=(0.2, 0.28)),
    "agentic_bf16_v151936": dict(
        T=65536, V=V_QWEN3, dtype=torch.bfloat16, z_std=3.0, peak=8.0, heavy_frac=0.0,
        heavy_peak=0.0, old_std=0.2, mu=("normal", 0.02), adv=("grpo", 0.3, 8),
        layout=("packed", 128, 64, 1024), band=(0.8, 1.25), eps=(0.2, 0.28)),
    # The thresholds of the paper's snapshot runs (App. D, run snap1004_1003: band
    # [1/1.004, 1.004], clip 0.003 on both sides), with old-policy and rollout
    # noise small enough that both ratios straddle them; float32 logits, since a
    # bf16 logit step (2^-6 at |z| ~ 3) is coarser than the thresholds; per-token
    # N(0, 1) advantages of both signs, so every token carries a gradient.
    "tight_f32_v151936": dict(
        T=2048, V=V_QWEN3, dtype=torch.float32, z_std=3.0, peak=8.0, heavy_frac=0.0,
        heavy_peak=0.0, old_std=0.003, mu=("normal", 0.003), adv=("normal",),
        layout=("none",), band=(1.0 / 1.004, 1.004), eps=(0.003, 0.003)),
    "heavytail_bf16_v151936": dict(
        T=16384, V=V_QWEN3, dtype=torch.bfloat16, z_std=3.0, peak=8.0, heavy_frac=0.1,
        heavy_peak=20.0, old_std=0.2, mu=("t2", 0.1), adv=("normal",), layout=("none",),
        band=(0.5, 2.0), eps=(0.2, 0.28)),
}


@dataclass
class LossBatch:
    name: str
    z_theta: torch.Tensor      # [T, V] current-policy logits
    z_old: torch.Tensor        # [T, V] old / proxy-policy logits
    ids: torch.Tensor          # [T] int32 sampled tokens
    logp_mu: torch.Tensor      # [T] float32 inference-side log-probabilities
    adv: torch.Tensor          # [T] float32 advantages
    mask: torch.Tensor = None  # [T] uint8 loss mask, or None (all tokens count)
    rd_lo: float = 0.5
    rd_hi: float = 2.0
    eps_low: float = 0.2
    eps_high: float = 0.28
    meta: dict = field(default_factory=dict)

    @property
    def T(self):
        return self.z_theta.shape[0]

    @property
    def V(self):
        return self.z_theta.shape[1]

    def thresholds(self):
        return dict(rd_lo=self.rd_lo, rd_hi=self.rd_hi, eps_low=self.eps_low,
                    eps_high=self.eps_high)


def _grpo_advantages(rng, n_seq, p, group):
    """Per-sequence advantages: Bernoulli(p) rewards normalised within groups
    of consecutive sequences, A = (R - mean) / (std + 1e-6), population std."""
    R = (rng.random(n_seq) < p).astype(np.float64)
    A = np.zeros(n_seq)
    for g0 in range(0, n_seq, group):
        r = R[g0:g0 + group]
        A[g0:g0 + group] = (r - r.mean()) / (r.std() + 1e-6)
    return A


def _sequence_layout(spec, rng, T):
    """Token -> (advantage, mask) from the workload's sequence structure."""
    kind = spec["layout"][0]
    adv = np.zeros(T, dtype=np.float32)
    mask = None
    if kind == "fixed":
        # a batch resized below the workload's T keeps its number of sequences
        # (shorter ones), so that its GRPO groups still have spread advantages
        L = spec["layout"][1]
        if T < spec["T"]:
            L = max(1, (L * T) // spec["T"])
        n_seq = (T + L - 1) // L
        A = _grpo_advantages(rng, n_seq, spec["adv"][1], spec["adv"][2])
        adv[:] = np.repeat(A, L)[:T]
    elif kind == "packed":
        n_seq, lo, hi = spec["layout"][1:]
        lengths = rng.integers(lo, hi + 1, size=n_seq)
        prompts = np.array([rng.integers(0, L // 4 + 1) for L in lengths])
        A = _grpo_advantages(rng, n_seq, spec["adv"][1], spec["adv"][2])
        mask = np.zeros(T, dtype=np.uint8)
        pos = 0
        for L, P, a in zip(lengths, prompts, A):
            if pos >= T:
                break
            end = min(T, pos + L)
            adv[pos:end] = a
            mask[min(T, pos + P):end] = 1
            pos = end
    else:  # per-token N(0, 1) advantages, every token counts
        adv[:] = rng.standard_normal(T)
    return adv, mask


def make_loss_batch(name, T=None, V=None, seed=0, device="cpu", chunk=1024):
    """Builds one seeded batch of the named workload (optionally resized)."""
    spec = dict(WORKLOADS[name])
    T = spec["T"] if T is None else int(T)
    V = spec["V"] if V is None else int(V)
    dev = torch.device(device)
    rng = np.random.default_rng(seed)
    adv, mask = _sequence_layout(spec, rng, T)
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    z = torch.empty((T, V), dtype=spec["dtype"], device=dev)
    zo = torch.empty((T, V), dtype=spec["dtype"], device=dev)
    ids = torch.empty(T, dtype=torch.int32, device=dev)
    lmu = torch.empty(T, dtype=torch.float32, device=dev)
    for r0 in range(0, T, chunk):
        r1 = min(T, r0 + chunk)
        n = r1 - r0
        x = torch.randn((n, V), generator=g, device=dev) * spec["z_std"]
        if spec["peak"] or spec["heavy_peak"]:
            pid = torch.randint(0, V, (n,), generator=g, device=dev)
            heavy = torch.rand(n, generator=g, device=dev) < spec["heavy_frac"]
            bump = torch.where(heavy, torch.full((n,), spec["heavy_peak"], device=dev),
                               torch.full((n,), spec["peak"], device=dev))
            x[torch.arange(n, device=dev), pid] += bump
        xo = x + torch.randn((n, V), generator=g, device=dev) * spec["old_std"]
        z[r0:r1] = x.to(spec["dtype"])
        zo[r0:r1] = xo.to(spec["dtype"])
        del x, xo
        # rollout engine emulation: sample from the old policy, report its logprob + noise
        zof = zo[r0:r1].float()
        u = torch.rand((n, V), generator=g, device=dev).clamp_(min=1e-30)
        y = torch.argmax(zof - torch.log(-torch.log(u)), dim=1)
        del u
        lp = torch.log_softmax(zof, dim=1).gather(1, y[:, None])[:, 0]
        del zof
        kind, scale = spec["mu"]
        noise = torch.randn(n, generator=g, device=dev)
        if kind == "t2":  # Student-t, 2 degrees of freedom: Z / sqrt(chi2_2 / 2)
            w = torch.rand(n, generator=g, device=dev).clamp_(min=1e-30)
            noise = noise / torch.sqrt(-torch.log(w))
        ids[r0:r1] = y.to(torch.int32)
        lmu[r0:r1] = lp + scale * noise
    return LossBatch(
        name=name, z_theta=z, z_old=zo, ids=ids, logp_mu=lmu,
        adv=torch.from_numpy(adv).to(dev),
        mask=None if mask is None else torch.from_numpy(mask).to(dev),
        rd_lo=spec["band"][0], rd_hi=spec["band"][1], eps_low=spec["eps"][0],
        eps_high=spec["eps"][1], meta=dict(seed=seed, workload=name, T=T, V=V))


def make_ewma_buffers(n, seed=0, device="cpu", chunk=1 << 26):
    """theta ~ N(0, 0.02^2) and theta_prox = theta + N(0, 1e-4^2), float32 [n]."""
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    theta = torch.empty(n, dtype=torch.float32, device=dev)
    prox = torch.empty(n, dtype=torch.float32, device=dev)
    for i0 in range(0, n, chunk):
        i1 = min(n, i0 + chunk)
        t = torch.randn(i1 - i0, generator=g, device=dev) * 0.02
        theta[i0:i1] = t
        prox[i0:i1] = t + torch.randn(i1 - i0, generator=g, device=dev) * 1e-4
    return theta, prox
