"""Seeded synthetic inputs for the ACRL hot path.

This module is shared by the tests, the smoke check and the benchmark; it
feeds the CUDA path and the float64 oracle the SAME materialised buffers.  It
holds none of the method's own arithmetic (no log-softmax statistics of pi,
no discrepancy, weight, advantage or gradient).  What it does compute stands
in for the two engines that produce the method's inputs:

  * pi's logits: synthetic bf16 rows with the distribution each workload names;
  * the sampled token ids: drawn from softmax(pi) by the Gumbel-max trick;
  * mu's cached log-probs: what an FP8-E4M3 rollout engine reports, emulated by
    quantising pi's logits to E4M3 (nearest-even, or truncation toward zero as
    in the stress test of Sec. 5.3), then torch's own log_softmax, plus noise;
  * rewards: Bernoulli draws per response.

Structure (lengths, rewards, which sequences get an extra perturbation) comes
from a CPU generator so that it is identical on every device; element data
comes from a generator on the target device.
"""

from __future__ import annotations

from dataclasses import dataclass, replace

import torch

E4M3_MAX = 448.0


@dataclass(frozen=True)
class WorkloadSpec:
    name: str
    n_prompts: int           # Q: prompts in the batch
    group_size: int          # G: responses per prompt
    len_lo: int              # response length ~ U{len_lo .. len_hi}
    len_hi: int
    V: int                   # vocabulary size
    dist: str = "normal"     # "normal" | "student_t"
    scale: float = 2.0       # std of the normal, or scale of the Student-t
    dof: float = 4.0         # Student-t degrees of freedom
    boost_frac: float = 0.0  # fraction of each row's entries raised by `boost`
    boost: float = 0.0
    pad_multiple: int = 0    # right-pad each response to a multiple (mask 0)
    fp8_scale: str = "row"   # "row" (per token) or "tensor"
    fp8_round: str = "nearest"  # "nearest" or "trunc"
    mu_noise: float = 0.0    # N(0, mu_noise^2) added to mu's log-probs
    perturb_frac: float = 0.0  # fraction of responses with an extra perturbation
    perturb_std: float = 0.0
    reward_p: float = 0.5    # Bernoulli reward probability
    chunk_rows: int = 0      # rows per chunk for the long workload (0 = one chunk)
    ld_pad: int = 0          # extra columns beyond V rounded up to 8

    @property
    def ld(self) -> int:
        return ((self.V + 7) // 8) * 8 + self.ld_pad

    @property
    def n_seqs(self) -> int:
        return self.n_prompts * self.group_size


# The five workloads: shapes and distributions of the paper's settings
# (batch of prompts x n responses, response lengths up to 2048 / 8192+,
# Qwen2.5 vocabulary of 151,936, FP8 rollout).
TINY = WorkloadSpec("tiny", 4, 1, 256, 256, 4096, dist="normal", scale=2.0,
                    fp8_scale="row", mu_noise=0.01, reward_p=0.5)
GRPO = WorkloadSpec("grpo", 8, 8, 64, 1024, 32000, dist="normal", scale=3.0, boost_frac=0.01,
                    boost=8.0, pad_multiple=64, fp8_scale="tensor", mu_noise=0.02, reward_p=0.3)
QWEN = WorkloadSpec("qwen", 16, 8, 256, 2048, 151936, dist="student_t", scale=2.0, dof=4.0,
                    fp8_scale="tensor", perturb_frac=0.1, perturb_std=0.3, reward_p=0.3)
LONG = WorkloadSpec("long", 8, 4, 4096, 16384, 151936, dist="normal", scale=2.0,
                    fp8_scale="tensor", reward_p=0.3, chunk_rows=65536)

# The Qwen workload at 8,192 rows (2.5 GB of logits): small enough for a full
# profiler capture, still far larger than L2.
QWEN_PROFILE = replace(QWEN, name="qwen_profile", n_prompts=2, group_size=4, len_lo=1024, len_hi=1024)

# The batch of the paper's overhead measurement (Sec. 5.4 on the App. A 3B
# setting: 64 prompts x 8 responses, responses up to 2048 tokens), for the
# weight calls alone (token-level inputs, no logits).
WEIGHTS_SEC54 = WorkloadSpec("weights_sec54", 64, 8, 1, 2048, 151936, reward_p=0.3, perturb_frac=0.1,
                             perturb_std=0.3)

SPECS = {s.name: s for s in (TINY, GRPO, QWEN, LONG, QWEN_PROFILE)}
BASE_SEED = 2607_24062


def seed_for(name: str, step: int = 0) -> int:
    order = ["tiny", "grpo", "qwen", "long", "lmhead"]
    k = order.index(name) if name in order else 7
    return BASE_SEED + k + 1000 * step


# --------------------------------------------------------------------------
# structure
# --------------------------------------------------------------------------

@dataclass
class Structure:
    lengths: torch.Tensor        # int64 [S] valid tokens per response
    seq_offsets: torch.Tensor    # int64 [S+1] row offsets (padding included)
    group_offsets: torch.Tensor  # int32 [Q+1] sequence offsets per prompt
    mask: torch.Tensor           # uint8 [T]
    rewards: torch.Tensor        # float32 [S]
    perturbed: torch.Tensor      # bool [S]
    T: int


def make_structure(spec: WorkloadSpec, seed: int) -> Structure:
    g = torch.Generator().manual_seed(seed)
    S = spec.n_seqs
    lengths = torch.randint(spec.len_lo, spec.len_hi + 1, (S,), generator=g, dtype=torch.int64)
    if spec.pad_multiple:
        rows = (lengths + spec.pad_multiple - 1) // spec.pad_multiple * spec.pad_multiple
    else:
        rows = lengths.clone()
    seq_offsets = torch.zeros(S + 1, dtype=torch.int64)
    seq_offsets[1:] = torch.cumsum(rows, 0)
    T = int(seq_offsets[-1])
    mask = torch.zeros(T, dtype=torch.uint8)
    for i in range(S):
        mask[seq_offsets[i]: seq_offsets[i] + lengths[i]] = 1
    group_offsets = (torch.arange(spec.n_prompts + 1, dtype=torch.int64) * spec.group_size).to(torch.int32)
    rewards = (torch.rand(S, generator=g) < spec.reward_p).to(torch.float32)
    perturbed = torch.rand(S, generator=g) < spec.perturb_frac
    return Structure(lengths, seq_offsets, group_offsets, mask, rewards, perturbed, T)


# --------------------------------------------------------------------------
# FP8-E4M3 emulation of the rollout engine's quantiser
# --------------------------------------------------------------------------

def e4m3_values() -> torch.Tensor:
    """All finite non-negative E4M3 (fn variant) values, ascending (float32)."""
    codes = torch.arange(0, 0x7F, dtype=torch.uint8)  # 0x7F is NaN in the fn variant
    return codes.view(torch.float8_e4m3fn).to(torch.float32)


def e4m3_roundtrip(y: torch.Tensor, rounding: str = "nearest") -> torch.Tensor:
    """Quantise float32 `y` (already divided by its scale) to E4M3 and back.
    "nearest": round to nearest, ties to even (the standard quantiser of
    Sec. 5.1); "trunc": toward zero, Q(x) = trunc(x/S) (Sec. 5.3)."""
    y = y.clamp(-E4M3_MAX, E4M3_MAX)
    if rounding == "nearest":
        return y.to(torch.float8_e4m3fn).to(torch.float32)
    if rounding == "trunc":
        grid = e4m3_values().to(y.device)
        mag = y.abs()
        idx = torch.searchsorted(grid, mag.contiguous(), right=True) - 1
        return torch.copysign(grid[idx.clamp_min(0)], y)
    raise ValueError(rounding)


# --------------------------------------------------------------------------
# element data
# --------------------------------------------------------------------------

@dataclass
class Batch:
    spec: WorkloadSpec
    seed: int
    logits: torch.Tensor         # bf16 [T, ld] (columns >= V are zero)
    ids: torch.Tensor            # int32 [T]
    mask: torch.Tensor           # uint8 [T]
    logp_mu: torch.Tensor        # float32 [T]
    rewards: torch.Tensor        # float32 [S]
    seq_offsets: torch.Tensor    # int64 [S+1]
    group_offsets: torch.Tensor  # int32 [Q+1]
    T: int

    @property
    def V(self) -> int:
        return self.spec.V

    @property
    def ld(self) -> int:
        return self.spec.ld

    @property
    def S(self) -> int:
        return self.seq_offsets.numel() - 1

    @property
    def Gn(self) -> int:
        return self.group_offsets.numel() - 1


def _fill_logits(spec: WorkloadSpec, out: torch.Tensor, gen: torch.Generator, rows_per_chunk: int):
    T, V = out.shape[0], spec.V
    dev = out.device
    for r0 in range(0, T, rows_per_chunk):
        r1 = min(T, r0 + rows_per_chunk)
        n = r1 - r0
        if spec.dist == "normal":
            z = torch.randn((n, V), generator=gen, device=dev) * spec.scale
        elif spec.dist == "student_t":
            # t_nu = N / sqrt(chi2_nu / nu), chi2_nu a sum of nu squared normals (nu integer)
            k = int(spec.dof)
            num = torch.randn((n, V), generator=gen, device=dev)
            chi2 = torch.zeros((n, V), device=dev)
            for _ in range(k):
                e = torch.randn((n, V), generator=gen, device=dev)
                chi2.addcmul_(e, e)
            z = num * torch.rsqrt(chi2 / k) * spec.scale
            del num, chi2
        else:
            raise ValueError(spec.dist)
        if spec.boost_frac > 0:
            hit = torch.rand((n, V), generator=gen, device=dev) < spec.boost_frac
            z += hit.to(z.dtype) * spec.boost
            del hit
        out[r0:r1, :V] = z.to(torch.bfloat16)
        del z


def _sample_and_mu(spec: WorkloadSpec, logits: torch.Tensor, gen: torch.Generator,
                   rows_per_chunk: int, tensor_scale: float | None):
    T, V = logits.shape[0], spec.V
    dev = logits.device
    ids = torch.empty(T, dtype=torch.int32, device=dev)
    logp_mu = torch.empty(T, dtype=torch.float32, device=dev)
    for r0 in range(0, T, rows_per_chunk):
        r1 = min(T, r0 + rows_per_chunk)
        z = logits[r0:r1, :V].to(torch.float32)
        # a_t ~ softmax(pi): Gumbel-max
        u = torch.rand(z.shape, generator=gen, device=dev)
        a = torch.argmax(z - torch.log(-torch.log(u)), dim=1)
        del u
        ids[r0:r1] = a.to(torch.int32)
        # mu: the rollout engine's FP8-E4M3 view of the same logits
        if tensor_scale is None:
            s = (z.abs().amax(dim=1, keepdim=True) / E4M3_MAX).clamp_min(1e-30)
        else:
            s = torch.tensor(tensor_scale, dtype=torch.float32, device=dev)
        zq = e4m3_roundtrip(z / s, spec.fp8_round) * s
        del z
        lsm = torch.log_softmax(zq, dim=1)
        logp_mu[r0:r1] = lsm.gather(1, a.view(-1, 1)).view(-1)
        del zq, lsm
    return ids, logp_mu


def _chunk_rows(spec: WorkloadSpec, budget_elems: int) -> int:
    return max(1, min(65536, budget_elems // max(1, spec.V)))


def generate(spec: WorkloadSpec, seed: int | None = None, device="cpu",
             budget_elems: int = 1 << 28) -> Batch:
    """Materialise one batch of `spec` on `device`."""
    if seed is None:
        seed = seed_for(spec.name)
    st = make_structure(spec, seed)
    dev = torch.device(device)
    gen = torch.Generator(device=dev).manual_seed(seed + 17)
    rows = _chunk_rows(spec, budget_elems)
    logits = torch.zeros((st.T, spec.ld), dtype=torch.bfloat16, device=dev)
    _fill_logits(spec, logits, gen, rows)
    tensor_scale = None
    if spec.fp8_scale == "tensor":
        amax = 0.0
        for r0 in range(0, st.T, rows):
            amax = max(amax, float(logits[r0:r0 + rows, :spec.V].abs().max().float()))
        tensor_scale = max(amax, 1e-30) / E4M3_MAX
    ids, logp_mu = _sample_and_mu(spec, logits, gen, rows, tensor_scale)
    if spec.mu_noise > 0:
        logp_mu += torch.randn(st.T, generator=gen, device=dev) * spec.mu_noise
    if spec.perturb_frac > 0:
        noise = torch.randn(st.T, generator=gen, device=dev) * spec.perturb_std
        per_row = torch.repeat_interleave(st.perturbed, st.seq_offsets[1:] - st.seq_offsets[:-1]).to(dev)
        logp_mu += noise * per_row.to(noise.dtype)
    logp_mu.clamp_(max=0.0)
    return Batch(spec, seed, logits, ids, st.mask.to(dev), logp_mu, st.rewards.to(dev),
                 st.seq_offsets.to(dev), st.group_offsets.to(dev), st.T)


# --------------------------------------------------------------------------
# fused LM-head workload: hidden states and the LM-head weight
# --------------------------------------------------------------------------

@dataclass
class LMHeadBatch:
    hidden: torch.Tensor         # bf16 [T, K] ~ N(0, 1)
    weight: torch.Tensor         # bf16 [N, K] ~ N(0, w_std^2)
    ids: torch.Tensor            # int32 [T]
    mask: torch.Tensor           # uint8 [T]
    logp_mu: torch.Tensor        # float32 [T]
    rewards: torch.Tensor        # float32 [S]
    seq_offsets: torch.Tensor    # int64 [S+1]
    group_offsets: torch.Tensor  # int32 [Q+1]
    T: int
    N: int
    K: int

    @property
    def S(self) -> int:
        return self.seq_offsets.numel() - 1

    @property
    def Gn(self) -> int:
        return self.group_offsets.numel() - 1


LMHEAD = WorkloadSpec("lmhead", 16, 8, 256, 256, 151936, dist="normal", fp8_scale="row", reward_p=0.3)
LMHEAD_K = 4096
LMHEAD_W_STD = 0.02


def _rowwise_e4m3(x: torch.Tensor) -> torch.Tensor:
    s = (x.abs().amax(dim=1, keepdim=True) / E4M3_MAX).clamp_min(1e-30)
    return e4m3_roundtrip(x / s, "nearest") * s


def generate_lmhead(spec: WorkloadSpec = LMHEAD, K: int = LMHEAD_K, w_std: float = LMHEAD_W_STD,
                    seed: int | None = None, device="cpu", rows_per_chunk: int = 2048) -> LMHeadBatch:
    """Hidden states H ~ N(0,1) and weight W ~ N(0, w_std^2) in bf16.  The
    sampled ids come from softmax(H W^T) by Gumbel-max; mu's log-probs from the
    rollout engine's FP8 view: H quantised per token and W per output channel
    to E4M3 (Sec. 5.1), multiplied, log-softmax at the sampled id.  The
    products here are torch library matmuls standing in for the two engines."""
    if seed is None:
        seed = seed_for("lmhead")
    st = make_structure(spec, seed)
    dev = torch.device(device)
    gen = torch.Generator(device=dev).manual_seed(seed + 17)
    T, N = st.T, spec.V
    hidden = torch.randn((T, K), generator=gen, device=dev).to(torch.bfloat16)
    weight = (torch.randn((N, K), generator=gen, device=dev) * w_std).to(torch.bfloat16)
    cdt = torch.float32 if dev.type == "cpu" else torch.bfloat16
    wq = torch.empty_like(weight)
    for r0 in range(0, N, 8192):
        wq[r0:r0 + 8192] = _rowwise_e4m3(weight[r0:r0 + 8192].float()).to(torch.bfloat16)
    ids = torch.empty(T, dtype=torch.int32, device=dev)
    logp_mu = torch.empty(T, dtype=torch.float32, device=dev)
    for r0 in range(0, T, rows_per_chunk):
        r1 = min(T, r0 + rows_per_chunk)
        z = (hidden[r0:r1].to(cdt) @ weight.to(cdt).T).float()
        u = torch.rand(z.shape, generator=gen, device=dev)
        a = torch.argmax(z - torch.log(-torch.log(u)), dim=1)
        del u, z
        ids[r0:r1] = a.to(torch.int32)
        hq = _rowwise_e4m3(hidden[r0:r1].float()).to(cdt)
        zq = (hq @ wq.to(cdt).T).float()
        logp_mu[r0:r1] = torch.log_softmax(zq, dim=1).gather(1, a.view(-1, 1)).view(-1)
        del zq, hq
    logp_mu.clamp_(max=0.0)
    return LMHeadBatch(hidden, weight, ids, st.mask.to(dev), logp_mu, st.rewards.to(dev), st.seq_offsets.to(dev),
                       st.group_offsets.to(dev), T, N, K)


def small_variant(spec: WorkloadSpec, **kw) -> WorkloadSpec:
    """Same distributions at a size the oracle finishes in seconds."""
    return replace(spec, **kw)


def token_level(spec: WorkloadSpec, seed: int, device="cpu"):
    """O(T) inputs only (no logits): pi_old log-probs, mu log-probs, mask,
    rewards and offsets, for multi-step controller trajectories.  pi's
    log-probs are -2 * Exp(1) draws; mu's are pi's plus N(0, 0.02^2) (plus the
    spec's perturbation), clamped to <= 0."""
    st = make_structure(spec, seed)
    dev = torch.device(device)
    gen = torch.Generator().manual_seed(seed + 29)
    logp_pi = -2.0 * torch.empty(st.T).exponential_(1.0, generator=gen)
    logp_mu = logp_pi + 0.02 * torch.randn(st.T, generator=gen)
    if spec.perturb_frac > 0:
        per_row = torch.repeat_interleave(st.perturbed, st.seq_offsets[1:] - st.seq_offsets[:-1])
        logp_mu += spec.perturb_std * torch.randn(st.T, generator=gen) * per_row.float()
    logp_mu.clamp_(max=0.0)
    return {
        "logp_pi": logp_pi.float().to(dev), "logp_mu": logp_mu.float().to(dev), "mask": st.mask.to(dev),
        "rewards": st.rewards.to(dev), "seq_offsets": st.seq_offsets.to(dev),
        "group_offsets": st.group_offsets.to(dev), "T": st.T,
    }


def expected_tokens(spec: WorkloadSpec) -> float:
    return spec.n_seqs * (spec.len_lo + spec.len_hi) / 2.0


def describe(spec: WorkloadSpec) -> str:
    return (f"{spec.name}: Q={spec.n_prompts} G={spec.group_size} len~U[{spec.len_lo},{spec.len_hi}] "
            f"V={spec.V} ld={spec.ld} {spec.dist}(scale={spec.scale}) fp8={spec.fp8_scale}/{spec.fp8_round}")


__all__ = ["WorkloadSpec", "TINY", "GRPO", "QWEN", "LONG", "LMHEAD", "WEIGHTS_SEC54", "SPECS", "generate", "make_structure",
           "generate_lmhead", "LMHeadBatch", "LMHEAD_K", "LMHEAD_W_STD",
           "e4m3_roundtrip", "e4m3_values", "seed_for", "small_variant", "token_level", "Batch",
           "expected_tokens", "describe", "E4M3_MAX"]

