"""Seeded gradient vectors for a workload.

Seeds: numpy PCG64 streams from SeedSequence entropy
  [BASE_SEED, config id, 0xB10C]               per-block scales (once per configuration)
  [BASE_SEED, config id, 0x5111E]              spike positions and signs (once per config)
  [BASE_SEED, config id, step, worker]         the entries of one worker's gradient
  [BASE_SEED, config id, step, worker, 1]      Laplace signs of those entries
Every stream is consumed in coordinate order, so a draw of the first n coordinates equals
the first n coordinates of the full draw.
Spikes model persistent heavy coordinates: the same positions and signs for every worker
and step, added on top of the block noise.
"""

from __future__ import annotations

import numpy as np

from .configs import Workload

BASE_SEED = 20210813


def _rng(*words: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([BASE_SEED, *words])))


def block_scales(w: Workload) -> np.ndarray:
    """Per-block scale (sigma or Laplace b), log-uniform in [scale_lo, scale_hi]."""
    nb = len(w.blocks)
    if w.scale_lo == w.scale_hi:
        return np.full(nb, w.scale_lo, dtype=np.float64)
    u = _rng(w.cid, 0xB10C).random(nb)
    return np.exp(np.log(w.scale_lo) + u * (np.log(w.scale_hi) - np.log(w.scale_lo)))


def spike_positions(w: Workload):
    """(positions ascending int64, signs +-1 float32) of the spike coordinates."""
    n = int(round(w.spike_frac * w.d))
    if n == 0:
        return np.zeros(0, dtype=np.int64), np.zeros(0, dtype=np.float32)
    g = _rng(w.cid, 0x5111E)
    pos = np.sort(g.choice(w.d, size=n, replace=False)).astype(np.int64)
    sgn = np.where(g.random(n) < 0.5, -1.0, 1.0).astype(np.float32)
    return pos, sgn


def _scale_vector(w: Workload) -> np.ndarray:
    return np.repeat(block_scales(w).astype(np.float32), w.blocks)


def make_gradient(w: Workload, step: int, worker: int, out: np.ndarray | None = None,
                  d: int | None = None, _cache: dict = {}) -> np.ndarray:
    """Gradient of ``worker`` at ``step`` as fp32 [d] (optionally only the first d coords).

    Entries are N(0, s_l^2) or Laplace(0, b_l) per block l (Laplace drawn as a standard
    exponential times an independent random sign), plus the configuration's spikes.
    """
    n = w.d if d is None else d
    key = w.cid
    if key not in _cache:
        _cache.clear()
        _cache[key] = (_scale_vector(w), *spike_positions(w))
    scale, pos, sgn = _cache[key]
    g = _rng(w.cid, step, worker)
    if w.dist == "normal":
        x = g.standard_normal(n, dtype=np.float32)
    elif w.dist == "laplace":
        x = g.standard_exponential(n, dtype=np.float32)
        flip = _rng(w.cid, step, worker, 1).random(n, dtype=np.float32) < 0.5
        np.negative(x, out=x, where=flip)
    else:
        raise ValueError(w.dist)
    x *= scale[:n]
    if pos.size:
        m = pos < n
        x[pos[m]] += np.float32(w.spike_mag) * sgn[m]
    if out is not None:
        out[:] = x
        return out
    return x


def make_gradients(w: Workload, step: int, workers=None, d: int | None = None, threads: int = 8):
    """List of gradients for ``workers`` (default all P) at ``step``, generated in threads."""
    from concurrent.futures import ThreadPoolExecutor
    ws = list(range(w.P)) if workers is None else list(workers)
    make_gradient(w, step, ws[0], d=1)  # fill the per-config cache before threading
    with ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
        return list(ex.map(lambda p: make_gradient(w, step, p, d=d), ws))


def torch_seed(w: Workload, step: int, worker: int) -> int:
    """64-bit seed of a device-side draw for (workload, step, worker)."""
    ss = np.random.SeedSequence([BASE_SEED, w.cid, step, worker, 2])
    return int(ss.generate_state(1, dtype=np.uint64)[0] & np.uint64((1 << 63) - 1))


_DEVICE_SCALES: dict = {}


def _device_scales(w: Workload, device):
    """The per-coordinate block scales of ``w`` as an fp32 device vector (one per workload and
    device, kept between calls)."""
    import torch
    key = (w.name, w.d, w.cid, str(device))
    if key not in _DEVICE_SCALES:
        _DEVICE_SCALES.clear()
        _DEVICE_SCALES[key] = torch.from_numpy(_scale_vector(w)).to(device)
    return _DEVICE_SCALES[key]


def make_gradient_torch(w: Workload, step: int, worker: int, out):
    """Fill the fp32 device tensor ``out`` (length d) with a gradient of the same recipe as
    ``make_gradient``, drawn on the device by PyTorch's generator (a different stream of
    numbers from the numpy draw, the same distribution).  Used where host generation of
    hundreds of millions of entries per worker would dominate."""
    import torch
    gen = torch.Generator(device=out.device)
    gen.manual_seed(torch_seed(w, step, worker))
    if w.dist == "normal":
        out.normal_(0.0, 1.0, generator=gen)
    else:
        out.exponential_(1.0, generator=gen)
        flip = torch.empty_like(out).uniform_(0.0, 1.0, generator=gen) < 0.5
        torch.where(flip, -out, out, out=out)
        del flip
    out.mul_(_device_scales(w, out.device))
    pos, sgn = spike_positions(w)
    if pos.size:
        pt = torch.from_numpy(pos).to(out.device)
        out.index_add_(0, pt, torch.from_numpy(sgn * np.float32(w.spike_mag)).to(out.device))
    return out
