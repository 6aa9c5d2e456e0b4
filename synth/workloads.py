"""Workload shapes and seeded input draws for the BGPO LM-head ELBO path.

The paper trains LLaDA-8B-Instruct on math, code and planning data with response
lengths 512 / 256, G = 8 and n_t = 16 (Sec. 4.1, Table 5). Those datasets and
weights are not available here; these seeded synthetic inputs with the paper's
shapes stand in for them:

  * hidden states X ~ N(0, 1), LM head W ~ N(0, 1/H), both drawn in fp32 and
    rounded once to bf16 (round-to-nearest-even, by torch);
  * targets y^i uniform over V (tiny case) or truncated Zipf(s) over token ranks
    1..V, token id = rank - 1 (inverse CDF over the finite support);
  * advantages either drawn N(0, 1) directly, or produced from Bernoulli(0.5)
    rewards (the normalisation of Eq. 18 is done by each implementation, not here);
  * old-policy perturbation eps ~ N(0, 0.1^2) per (sequence, MC sample): each
    implementation forms its own l_old = l_self + eps (on-policy workloads use
    eps = 0, exercising the Equivalence property of Sec. 3.2).

Nothing here computes a step of the method.
"""
from dataclasses import dataclass, field, replace

import numpy as np


@dataclass(frozen=True)
class Workload:
    name: str
    B: int            # responses in the batch
    P: int            # prompt length
    R: int            # response length
    H: int            # hidden size
    V: int            # vocabulary size
    n_t: int          # MC samples per response
    G: int            # group size (Eq. 18; loss_scale = 1/G)
    t_mode: int       # 0 = t iid U(0,1], 1 = stratified over the n_t samples
    seed: int
    targets: str = "uniform"      # "uniform" or "zipf"
    zipf_s: float = 1.1
    advantages: str = "normal"    # "normal" (A ~ N(0,1)) or "bernoulli" (rewards)
    eps_std: float = 0.1          # 0.0 = on-policy
    note: str = ""

    @property
    def masked_rows_cap(self):
        return self.B * self.R

    def with_(self, **kw):
        return replace(self, **kw)


CONFIGS = {
    # parity-only case the oracle finishes in well under a second
    "tiny": Workload("tiny", B=2, P=16, R=32, H=64, V=512, n_t=4, G=2, t_mode=0, seed=1,
                     targets="uniform", advantages="normal", eps_std=0.1),
    # LLaDA-8B-shaped head, one group of 8, response 256
    "llada8b_r256": Workload("llada8b_r256", B=8, P=128, R=256, H=4096, V=126464, n_t=8, G=8,
                             t_mode=0, seed=2, targets="zipf", zipf_s=1.1,
                             advantages="bernoulli", eps_std=0.1),
    # same head, 16 responses of 512, stratified t, on-policy (Equivalence)
    "llada8b_r512_onpolicy": Workload("llada8b_r512_onpolicy", B=16, P=256, R=512, H=4096,
                                      V=126464, n_t=16, G=8, t_mode=1, seed=3,
                                      targets="zipf", zipf_s=1.1, advantages="bernoulli",
                                      eps_std=0.0),
    # half of the batch above: the small case for full ncu captures (~4.5 GB on device)
    "llada8b_r512_b8": Workload("llada8b_r512_b8", B=8, P=256, R=512, H=4096, V=126464, n_t=16,
                                G=8, t_mode=1, seed=6, targets="zipf", zipf_s=1.1,
                                advantages="bernoulli", eps_std=0.0),
    # n_t sweep (n_t overridden per point)
    "llada8b_sweep": Workload("llada8b_sweep", B=8, P=256, R=512, H=4096, V=126464, n_t=1, G=8,
                              t_mode=0, seed=4, targets="zipf", zipf_s=1.1,
                              advantages="bernoulli", eps_std=0.1),
    # Dream-7B-shaped head
    "dream7b": Workload("dream7b", B=32, P=512, R=1024, H=3584, V=152064, n_t=16, G=8, t_mode=0,
                        seed=5, targets="zipf", zipf_s=1.2, advantages="bernoulli",
                        eps_std=0.1),
    # parity cases spanning several tiles with ragged tails in every dimension
    # (advantages drawn directly: one group of 3 Bernoulli rewards can be all
    # equal, which makes every advantage, and every gradient, exactly zero)
    "ragged": Workload("ragged", B=3, P=5, R=301, H=192, V=1000, n_t=3, G=3, t_mode=0, seed=11,
                       targets="zipf", zipf_s=1.1, advantages="normal", eps_std=0.1),
    "ragged_strat": Workload("ragged_strat", B=5, P=3, R=130, H=320, V=777, n_t=5, G=5,
                             t_mode=1, seed=12, targets="uniform", advantages="normal",
                             eps_std=0.3),
}

SWEEP_NT = (1, 2, 4, 8, 16, 32)


def zipf_targets(rng, shape, V, s):
    """Token ids with P(id = k - 1) proportional to k^-s for k = 1..V (inverse CDF)."""
    ranks = np.arange(1, V + 1, dtype=np.float64)
    cdf = np.cumsum(ranks ** (-s))
    cdf /= cdf[-1]
    u = rng.random(size=shape)
    idx = np.searchsorted(cdf, u, side="right")
    return np.minimum(idx, V - 1).astype(np.int32)


def make_inputs(wl, device="cpu", need_w=True):
    """Seeded inputs of workload ``wl`` as torch tensors.

    Returns a dict with
      X        [B, P+R, H] bf16
      W        [V, H] bf16 (omitted when need_w is False)
      Y        [B, R] int32
      A        [B] fp32 (advantages="normal") or None
      rewards  [B] fp32 in {0, 1} (advantages="bernoulli") or None
      eps      [B, n_t] fp32 old-policy perturbation (zeros when on-policy)
    """
    import torch

    rng = np.random.default_rng(wl.seed)
    out = {}
    X = rng.standard_normal((wl.B, wl.P + wl.R, wl.H), dtype=np.float32)
    out["X"] = torch.from_numpy(X).to(torch.bfloat16)
    del X
    if wl.targets == "uniform":
        Y = rng.integers(0, wl.V, size=(wl.B, wl.R), dtype=np.int32)
    else:
        Y = zipf_targets(rng, (wl.B, wl.R), wl.V, wl.zipf_s)
    out["Y"] = torch.from_numpy(Y)
    if wl.advantages == "normal":
        out["A"] = torch.from_numpy(rng.standard_normal(wl.B).astype(np.float32))
        out["rewards"] = None
    else:
        out["A"] = None
        out["rewards"] = torch.from_numpy((rng.random(wl.B) < 0.5).astype(np.float32))
    eps = rng.standard_normal((wl.B, wl.n_t)).astype(np.float32) * np.float32(wl.eps_std)
    out["eps"] = torch.from_numpy(eps)
    if need_w:
        # W drawn from its own stream so that X/Y/A do not depend on V*H
        wrng = np.random.default_rng([wl.seed, 0x57])
        W = torch.empty((wl.V, wl.H), dtype=torch.bfloat16)
        scale = np.float32(1.0 / np.sqrt(wl.H))
        step = max(1, (1 << 24) // wl.H)
        for v0 in range(0, wl.V, step):
            v1 = min(wl.V, v0 + step)
            blk = wrng.standard_normal((v1 - v0, wl.H), dtype=np.float32) * scale
            W[v0:v1] = torch.from_numpy(blk).to(torch.bfloat16)
        out["W"] = W
    if device != "cpu":
        out = {k: (v.to(device) if v is not None else None) for k, v in out.items()}
    return out


def make_old_head(wl, W, delta=0.05):
    """An old-policy LM head W_old = W + delta * N(0, 1/H), rounded to bf16.

    Eq. 10 evaluates the current and the old policy on the same draws; a second
    head makes the two policies' l differ through the model rather than through
    a perturbation added to l. Seeded by (wl.seed, 0x01D); W is the bf16 head of
    make_inputs (CPU or device; the result lands on W's device).
    """
    import torch

    rng = np.random.default_rng([wl.seed, 0x01D])
    noise = rng.standard_normal((wl.V, wl.H), dtype=np.float32) * np.float32(delta / np.sqrt(wl.H))
    Wf = W.detach().to("cpu", torch.float32) + torch.from_numpy(noise)
    return Wf.to(torch.bfloat16).to(W.device)


def make_per_sample_hidden(wl, X, rho=0.8):
    """Final hidden states that differ between MC samples: X_j [n_t, B, P+R, H].

    In the paper each MC sample runs the network on its own masked sequence, so
    its hidden states differ (Sec. 2.1). X_j = rho X + sqrt(1 - rho^2) N(0, 1),
    drawn in fp32 from (wl.seed, 0x51, j) and rounded to bf16; X is the bf16
    tensor of make_inputs (the result lands on X's device).
    """
    import torch

    c = np.float32(np.sqrt(1.0 - rho * rho))
    Xf = X.detach().to("cpu", torch.float32)
    out = torch.empty((wl.n_t,) + tuple(X.shape), dtype=torch.bfloat16)
    for j in range(wl.n_t):
        rng = np.random.default_rng([wl.seed, 0x51, j])
        z = rng.standard_normal(tuple(X.shape), dtype=np.float32)
        out[j] = (Xf * np.float32(rho) + torch.from_numpy(z) * c).to(torch.bfloat16)
    return out.to(X.device)
