"""Seeded synthetic inputs shaped like the paper's hybrid-model layers.

This module is shared by the tests, the smoke check, the benchmark and the oracle harness.
It holds input synthesis only -- random draws and their fixed transforms (unit-norm keys,
softplus decay rates, sigmoid gates) -- and none of the method's arithmetic.

Layouts follow the library: per-token tensors are ``(B, T, H, d)`` float32, the per-head
gate ``beta`` and per-head decay rates are ``(B, T, H)``.

Two generators:

* :func:`host_inputs` -- numpy Philox, counter based: every ``(batch element, token)`` slice
  is drawn from its own key, so any sub-range of a huge workload can be regenerated without
  materialising the rest.  Used wherever the oracle must see the same numbers as the GPU.
* :func:`device_inputs` -- torch's CUDA generator, seeded; used by the benchmark to fill
  multi-gigabyte inputs directly in device memory.  Same distributions, different numbers.
"""
from __future__ import annotations

from dataclasses import dataclass, field
import numpy as np

# Families of Eq. (1) covered by the workloads.
KDA = "kda"        # per-row decay, delta-rule erase (a = beta k, w = beta 1)
GDN = "gdn"        # per-head decay, delta-rule erase
MAMBA2 = "mamba2"  # per-head decay, no erase (a = 0, w = 1)
KDA_GEN = "kda_general"   # per-row decay, a and w drawn per token (Eq. (1) in general)
GDN_GEN = "gdn_general"   # per-head decay, a and w drawn per token


@dataclass(frozen=True)
class Workload:
    """One synthetic layer workload (shapes, distributions and quantiser settings)."""
    name: str
    family: str
    B: int
    H: int
    dk: int
    dv: int
    T: int
    C: int
    bbar: int                 # mean payload bits per state element
    bmin: int
    bmax: int
    unit: str                 # "row" (width + scale per row) or "head" (width per head, block-32 scales)
    group_heads: int = 1      # heads per output-normalisation group (row unit)
    gate_bits: int = 0        # 0: FP32 decay rates; g > 0: log-quantised rates with 2**g levels
    s_loc: float = -2.0       # decay rate s = softplus(N(s_loc, 1))
    kq_std: float = 0.0       # 0: unit-norm Gaussian keys/queries; > 0: N(0, kq_std^2) entries
    persistent: float = 0.0   # > 0: per-channel decay fixed over tokens, log-uniform over
                              # [persistent, 1] (slow channels that keep their rate)
    seed: int = 0
    notes: str = field(default="", compare=False)

    @property
    def per_row_decay(self) -> bool:
        return self.family in (KDA, KDA_GEN)

    @property
    def erase(self) -> bool:
        return self.family != MAMBA2

    @property
    def general(self) -> bool:
        """a and w given per token instead of beta k and beta 1."""
        return self.family in (KDA_GEN, GDN_GEN)


# The five layer workloads: a tiny KDA recurrence, KDA decode, Gated DeltaNet decode,
# Mamba-2 decode and KDA prefill with chunked write-back.
WORKLOADS = {
    "tiny_kda": Workload("tiny_kda", KDA, B=1, H=1, dk=64, dv=64, T=256, C=1, bbar=2, bmin=1,
                         bmax=16, unit="row", seed=0),
    "kda_decode": Workload("kda_decode", KDA, B=256, H=32, dk=128, dv=128, T=1024, C=1, bbar=4,
                           bmin=0, bmax=8, unit="row", gate_bits=2, seed=1000),
    "gdn_decode": Workload("gdn_decode", GDN, B=64, H=16, dk=128, dv=128, T=2048, C=1, bbar=4,
                           bmin=2, bmax=16, unit="head", s_loc=-3.0, seed=2000),
    "mamba2_decode": Workload("mamba2_decode", MAMBA2, B=128, H=64, dk=128, dv=64, T=2048, C=1,
                              bbar=6, bmin=1, bmax=16, unit="row", group_heads=8, s_loc=-3.0,
                              kq_std=float(1.0 / np.sqrt(128.0)), seed=3000),
    "kda_prefill": Workload("kda_prefill", KDA, B=16, H=32, dk=128, dv=128, T=8192, C=64, bbar=3,
                            bmin=1, bmax=8, unit="row", seed=4000),
}

# Beyond the paper's layers: Eq. (1) with a and w given per token (a perturbed delta-rule
# erase vector, per-channel write gates).
EXTENSION_WORKLOADS = {
    "kda_general": Workload("kda_general", KDA_GEN, B=32, H=8, dk=128, dv=128, T=256, C=1, bbar=4,
                            bmin=1, bmax=8, unit="row", seed=5000),
    "gdn_general": Workload("gdn_general", GDN_GEN, B=16, H=16, dk=128, dv=128, T=256, C=1, bbar=4,
                            bmin=2, bmax=16, unit="head", s_loc=-3.0, seed=6000),
    # KDA with persistent per-channel decay: each (b, h, i) keeps one rate over all tokens,
    # log-uniform in [1e-3, 1] (slow channels accumulate errors across write-backs)
    "kda_persistent": Workload("kda_persistent", KDA, B=32, H=8, dk=128, dv=128, T=256, C=1,
                               bbar=4, bmin=0, bmax=8, unit="row", gate_bits=2, persistent=1e-3,
                               seed=7000),
}


def scaled(w: Workload, **changes) -> Workload:
    """A copy of ``w`` with some fields replaced (smaller test shapes of the same recipe)."""
    d = {f: getattr(w, f) for f in w.__dataclass_fields__}
    d.update(changes)
    return Workload(**d)


def _softplus(z: np.ndarray) -> np.ndarray:
    return np.logaddexp(0.0, z)


def _sigmoid(z: np.ndarray) -> np.ndarray:
    return 1.0 / (1.0 + np.exp(-z))


# stream ids inside one workload seed
_Q, _K, _V, _S, _BETA, _A, _W = 1, 2, 3, 4, 5, 6, 7


def _rng(seed: int, stream: int, b: int, t: int) -> np.random.Generator:
    key = np.array([(seed << 8) | stream, (b << 32) | t], dtype=np.uint64)
    return np.random.Generator(np.random.Philox(key=key))


def _keys(rng, H, d, std):
    g = rng.standard_normal((H, d))
    if std > 0:
        return g * std
    return g / np.linalg.norm(g, axis=-1, keepdims=True)


def host_inputs(w: Workload, b_range=None, t_range=None) -> dict:
    """Inputs for batch elements ``b_range`` and tokens ``t_range`` (host float32 arrays).

    Returns ``q, k, v`` of shape ``(nb, nt, H, d)``, ``s`` of shape ``(nb, nt, H, dk)`` for
    per-row decay or ``(nb, nt, H)`` for per-head decay, and ``beta`` ``(nb, nt, H)``.
    Slice ``(b, t)`` depends only on ``(w.seed, b, t)``.
    """
    b0, b1 = b_range if b_range is not None else (0, w.B)
    t0, t1 = t_range if t_range is not None else (0, w.T)
    nb, nt = b1 - b0, t1 - t0
    H, dk, dv = w.H, w.dk, w.dv
    q = np.empty((nb, nt, H, dk), np.float32)
    k = np.empty((nb, nt, H, dk), np.float32)
    v = np.empty((nb, nt, H, dv), np.float32)
    s = np.empty((nb, nt, H, dk) if w.per_row_decay else (nb, nt, H), np.float32)
    beta = np.empty((nb, nt, H), np.float32)
    if w.general:
        a = np.empty((nb, nt, H, dk), np.float32)
        wg = np.empty((nb, nt, H, dv), np.float32)
    for bi in range(nb):
        for ti in range(nt):
            b, t = b0 + bi, t0 + ti
            q[bi, ti] = _keys(_rng(w.seed, _Q, b, t), H, dk, w.kq_std)
            k[bi, ti] = _keys(_rng(w.seed, _K, b, t), H, dk, w.kq_std)
            v[bi, ti] = _rng(w.seed, _V, b, t).standard_normal((H, dv))
            shape = (H, dk) if w.per_row_decay else (H,)
            if w.persistent > 0:   # one draw per (b, channel), the same for every token
                u = _rng(w.seed, _S, b, 0).uniform(size=shape)
                s[bi, ti] = np.exp(np.log(w.persistent) * (1.0 - u))
            else:
                s[bi, ti] = _softplus(w.s_loc + _rng(w.seed, _S, b, t).standard_normal(shape))
            beta[bi, ti] = _sigmoid(_rng(w.seed, _BETA, b, t).standard_normal((H,)))
            if w.general:
                g = _rng(w.seed, _A, b, t).standard_normal((H, dk)) / np.sqrt(dk)
                a[bi, ti] = beta[bi, ti][:, None] * (k[bi, ti] + 0.1 * g)
                wg[bi, ti] = _sigmoid(_rng(w.seed, _W, b, t).standard_normal((H, dv)))
    out = dict(q=q, k=k, v=v, s=s, beta=beta)
    if w.general:
        out.update(a=a, w=wg)
    return out


def device_inputs(w: Workload, device="cuda", T=None, seed_offset=0):
    """Same distributions drawn on the device with torch's seeded CUDA generator."""
    import torch
    T = w.T if T is None else T
    gen = torch.Generator(device=device)
    gen.manual_seed(w.seed * 7919 + 17 + seed_offset)
    H, dk, dv, B = w.H, w.dk, w.dv, w.B
    f32 = dict(device=device, dtype=torch.float32, generator=gen)

    def keys(d):
        g = torch.randn((B, T, H, d), **f32)
        if w.kq_std > 0:
            return g.mul_(w.kq_std)
        return g.div_(torch.linalg.vector_norm(g, dim=-1, keepdim=True))

    q = keys(dk)
    k = keys(dk)
    v = torch.randn((B, T, H, dv), **f32)
    shape = (B, T, H, dk) if w.per_row_decay else (B, T, H)
    if w.persistent > 0:
        u = torch.rand((B, 1) + shape[2:], **f32)
        s = torch.exp(u.neg_().add_(1.0).mul_(float(np.log(w.persistent)))).expand(shape).contiguous()
    else:
        s = torch.nn.functional.softplus(torch.randn(shape, **f32).add_(w.s_loc))
    beta = torch.sigmoid(torch.randn((B, T, H), **f32))
    out = dict(q=q, k=k, v=v, s=s, beta=beta)
    if w.general:
        g = torch.randn((B, T, H, dk), **f32).div_(dk ** 0.5)
        out["a"] = beta[..., None] * (k + 0.1 * g)
        out["w"] = torch.sigmoid(torch.randn((B, T, H, dv), **f32))
    return out


def random_state(w: Workload, seed: int, scale: float = 1.0) -> np.ndarray:
    """A dense FP32 state ``(B, H, dk, dv)`` with row ranges spread over two decades."""
    rng = _rng(w.seed + seed, 9, 0, 0)
    x = rng.standard_normal((w.B, w.H, w.dk, w.dv))
    row_scale = np.exp(rng.uniform(np.log(0.1), np.log(10.0), size=(w.B, w.H, w.dk, 1)))
    return (x * row_scale * scale).astype(np.float32)
