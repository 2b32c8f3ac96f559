"""Seeded synthetic inputs for the OrderMoE hot path.

This module only draws random inputs; it holds none of the method's
arithmetic. Tests feed the same draws to the CUDA library and to the CPU
oracle; bench.py draws its workload here too.

Recipe (the shapes and value distributions of the paper's Mixtral-style MoE
layers and edge testbed, Section VI-A):
  * router rows: K cluster centroids ~ N(0, sigma^2) with sigma = 0.02; the
    row of expert e is centroid[e // (E / K)] + N(0, (noise_ratio * sigma)^2),
    noise_ratio = 0.25 (so same-cluster rows have cosine ~ 0.94, others ~ 0);
  * expert FFN weights W1, W3 [E, dff, d] and W2 [E, d, dff] ~ N(0, 0.02^2);
  * hidden states and calibration tokens ~ N(0, 1);
  * home server of each token: uniform over the M servers, or Zipf(1.1)
    (P(m) proportional to (m + 1)^-1.1);
  * server parameters drawn from the testbed's ranges: F_m ~ U[20, 110]
    TFLOP/s, B_{m,n} = B_{n,m} ~ U[1, 10] Gbit/s, tau_{m,n} = tau_{n,m} ~
    U[0.2, 20] ms; per-token transfer size z = 2 d bytes (a bf16 hidden
    state) and per-token expert work c = 6 d dff flop (three matmuls).
All values are drawn in fp32 with torch's generator and rounded to bf16
where the path takes bf16. The same seed on a different device gives
different values (CPU and CUDA generators differ); tests that compare with
the oracle draw on the CPU.
"""
from dataclasses import dataclass, replace

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    T: int            # tokens per layer call
    d: int            # model width
    E: int            # experts per layer
    k: int            # routed experts per token
    dff: int          # expert hidden width
    M: int            # logical servers
    n_clusters: int   # router clusters (similarity groups)
    theta: float      # similarity threshold of a single layer
    qbar: float       # per-token quality budget Qbar
    home: str = "uniform"   # or "zipf1.1"
    L: int = 1        # MoE layers
    steps: int = 1    # decode steps (decode stack only)
    sigma: float = 0.02
    noise_ratio: float = 0.25
    omega_T: float = 0.5
    omega_Q: float = 0.5
    n_cal: int = 4096          # calibration tokens for the similarity
    theta_min: float = 0.5
    theta_max: float = 0.9


WORKLOADS = {
    "tiny": Workload("tiny", T=64, d=256, E=8, k=2, dff=512, M=4, n_clusters=2, theta=0.5,
                     qbar=0.05),
    "mixtral_prefill": Workload("mixtral_prefill", T=4096, d=4096, E=8, k=2, dff=14336, M=4,
                                n_clusters=4, theta=0.5, qbar=0.05),
    "fine_grained": Workload("fine_grained", T=8192, d=2048, E=64, k=6, dff=1408, M=8,
                             n_clusters=8, theta=0.5, qbar=0.10, home="zipf1.1", n_cal=8192),
    "similarity": Workload("similarity", T=0, d=2048, E=64, k=6, dff=1408, M=8, n_clusters=8,
                           theta=0.5, qbar=0.10, L=24, n_cal=262144),
    "decode_stack": Workload("decode_stack", T=128, d=4096, E=8, k=2, dff=14336, M=4,
                             n_clusters=4, theta=0.5, qbar=0.5, L=32, steps=64),
}


def workload(name: str, **over) -> Workload:
    w = WORKLOADS[name]
    return replace(w, **over) if over else w


def _gen(seed: int, device="cpu") -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def normal(shape, std, seed, device="cpu", dtype=torch.bfloat16):
    g = _gen(seed, device)
    x = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x.to(dtype)


def router_weights(E, d, n_clusters, seed, sigma=0.02, noise_ratio=0.25, device="cpu"):
    """Clustered router rows [E, d] bf16; expert e belongs to cluster e // (E / K)."""
    assert E % n_clusters == 0
    cent = normal((n_clusters, d), sigma, seed, device, torch.float32)
    noise = normal((E, d), sigma * noise_ratio, seed + 7919, device, torch.float32)
    cluster = torch.arange(E, device=device) // (E // n_clusters)
    return (cent[cluster] + noise).to(torch.bfloat16)


def cluster_of(E, n_clusters):
    return np.arange(E) // (E // n_clusters)


def ffn_weights(E, d, dff, seed, std=0.02, device="cpu"):
    W1 = normal((E, dff, d), std, seed + 1, device)
    W3 = normal((E, dff, d), std, seed + 2, device)
    W2 = normal((E, d, dff), std, seed + 3, device)
    return W1, W3, W2


def hidden(T, d, seed, device="cpu"):
    return normal((T, d), 1.0, seed + 11, device)


def homes(T, M, seed, dist="uniform"):
    rng = np.random.default_rng(seed + 13)
    if dist == "uniform":
        return rng.integers(0, M, size=T).astype(np.uint8)
    if dist.startswith("zipf"):
        s = float(dist[4:])
        p = (np.arange(M) + 1.0) ** (-s)
        p /= p.sum()
        return rng.choice(M, size=T, p=p).astype(np.uint8)
    raise ValueError(dist)


def capacities(M, total_memory, ratio, seed):
    """Server memory C_m [M] f64 at a memory budget ratio (total capacity over
    the memory of one full copy of the experts, Section VI-G): heterogeneous,
    proportional to U[12, 48] (the testbed's GB range), scaled so that
    sum C = ratio * total_memory."""
    rng = np.random.default_rng(seed + 19)
    raw = rng.uniform(12.0, 48.0, size=M)
    return raw * (ratio * float(total_memory) / raw.sum())


def token_shares(home, M):
    """pi_m [M] f64: the share of the tokens whose home (user-server
    association) is server m, the estimate of Eq. 33's pi_m."""
    return np.bincount(np.asarray(home, dtype=np.int64), minlength=M)[:M] / float(len(home))


@dataclass
class ServerParams:
    F: np.ndarray      # [M] flop/s
    B: np.ndarray      # [M, M] bytes/s
    tau: np.ndarray    # [M, M] s
    z: float           # bytes per token transfer
    c: float           # flop per token per expert
    omega_T: float
    omega_Q: float


def server_params(M, d, dff, seed, omega_T=0.5, omega_Q=0.5):
    rng = np.random.default_rng(seed + 17)
    F = rng.uniform(20e12, 110e12, size=M)
    Bg = rng.uniform(1.0, 10.0, size=(M, M))
    tg = rng.uniform(0.2e-3, 20e-3, size=(M, M))
    B = np.triu(Bg, 1); B = B + B.T
    tau = np.triu(tg, 1); tau = tau + tau.T
    np.fill_diagonal(B, 1.0)     # unused: no transfer when s == m
    np.fill_diagonal(tau, 0.0)
    B = B * 1e9 / 8.0            # Gbit/s -> bytes/s
    return ServerParams(F=F, B=B, tau=tau, z=2.0 * d, c=6.0 * d * dff, omega_T=omega_T,
                        omega_Q=omega_Q)


def layer_inputs(w: Workload, seed=0, device="cpu", layer=0, with_ffn=True):
    """One MoE layer's synthetic inputs as torch tensors (bf16 where the path is bf16)."""
    s = seed + 1000 * layer
    out = {
        "X": hidden(w.T, w.d, s, device),
        "Wr": router_weights(w.E, w.d, w.n_clusters, s + 101, w.sigma, w.noise_ratio, device),
        "home": homes(w.T, w.M, s, w.home),
    }
    if with_ffn:
        out["W1"], out["W3"], out["W2"] = ffn_weights(w.E, w.d, w.dff, s + 202, device=device)
    return out


def calibration(n, d, seed, device="cpu"):
    """Calibration token representations for the similarity (Eq. 3), N(0, 1) bf16."""
    return normal((n, d), 1.0, seed + 29, device)


def bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> np.uint16 bit patterns (what the oracle takes)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def from_bits(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
