"""The five synthetic workloads of the benchmark plan, as data.

All use the cyclic assignment with N = m (Sec. III, Sec. IV).  Sizes:

  tiny      m=N=6,   delta=3,  d=64,      n_c=32,   least squares, fp32 X
  logistic  m=N=20,  delta=4,  d=4096,    n_c=512,  logistic, fp32 X ~ N(0,1)/sqrt(d)
  mse_sweep m=N=64,  delta=8,  d=65536,   n_c=1024, least squares, bf16 X ~ N(0,1)
  decode    m=N=256, delta=16, d=1048576, chunk gradients given, fp32 ~ N(0,1)
  sgd       m=N=128, delta=6,  d=8192,    n_c=2048, logistic, fp32 X ~ N(0,1)/sqrt(d)

Straggler models (psi_j = chunks processed by worker j, 0 <= psi_j <= delta):
  uniform      psi_j ~ U{0..delta}
  shifted_exp  per-chunk time tau_j = 1 + Exp(1) per worker; deadline
               T = 0.5 * delta * max_j tau_j (the slowest worker is half done);
               psi_j = min(delta, floor(T / tau_j))
  binomial     psi_j ~ Binomial(delta, p)
  frac_binom   f ~ U[0.2, 1] per pattern, psi_j ~ Binomial(delta, f)
"""
from __future__ import annotations

from dataclasses import dataclass, field


@dataclass(frozen=True)
class Config:
    name: str
    index: int
    N: int
    m: int
    delta: int
    d: int
    n_c: int              # points per chunk (0: chunk gradients are given)
    loss: str             # "lsq" | "logistic" | "none"
    x_dtype: str          # "f32" | "bf16" | "none"
    npat: int
    ells: tuple
    ell: int              # default communication factor
    pattern_model: str
    seed: int
    p_list: tuple = field(default=())
    iters: int = 0
    lr: float = 0.1

    @property
    def Ntil(self) -> int:
        return self.N * self.n_c


CONFIGS = {
    "tiny": Config("tiny", 0, N=6, m=6, delta=3, d=64, n_c=32, loss="lsq", x_dtype="f32",
                   npat=256, ells=(1, 2, 3), ell=2, pattern_model="uniform", seed=0),
    "logistic": Config("logistic", 1, N=20, m=20, delta=4, d=4096, n_c=512, loss="logistic",
                       x_dtype="f32", npat=10_000, ells=(1, 2, 4), ell=2,
                       pattern_model="shifted_exp", seed=1),
    "mse_sweep": Config("mse_sweep", 2, N=64, m=64, delta=8, d=65536, n_c=1024, loss="lsq",
                        x_dtype="bf16", npat=100_000, ells=(1, 2, 3), ell=2,
                        pattern_model="binomial", seed=2, p_list=(0.3, 0.5, 0.7)),
    "decode": Config("decode", 3, N=256, m=256, delta=16, d=1 << 20, n_c=0, loss="none",
                     x_dtype="none", npat=4096, ells=(1, 2, 4), ell=2,
                     pattern_model="frac_binom", seed=3),
    "sgd": Config("sgd", 4, N=128, m=128, delta=6, d=8192, n_c=2048, loss="logistic",
                  x_dtype="f32", npat=1, ells=(1, 2, 3), ell=2, pattern_model="shifted_exp",
                  seed=4, iters=64, lr=0.1),
}


def get(name: str) -> Config:
    return CONFIGS[name]
