"""Seeded synthetic session populations.

This module only draws random inputs; it holds none of the method's
arithmetic (no hashing, scoring, ranking, packing).  Both the CUDA path and
the CPU oracle consume what it produces, so both see identical bytes.

The populations stand in for the paper's three model classes (Table tab:pcs,
Sec. 7.2) -- Cosmos3-Nano's uint8 observation plus generator state,
WorldMem's growing memory bank, Matrix-Game 2.0's windowed paged KV context --
and for a mass suspend/resume under a host budget.  No model weights or
traces are used: every value is drawn from a seeded generator.

Sizes (configuration number in brackets):
  [1] markov      obs uint8 [3,256,256] ~ U{0..255}; rng {seed u64, offset u64}
  [2] banks       64 sessions, n ~ U[1,512]; key fp16[256] ~ N(0,1);
                  latent bf16[16,32,32] ~ N(0,1); query fp16[256]; k = min(n,128)
  [3] kv          256 sessions x 24 layers x 16 heads x 64, bf16 ~ N(0,1);
                  window 1024 tokens in 16-token pages, pages randomly
                  permuted in one global pool; ring start ~ U[0,1023]
  [4] classify    200 buffers, bytes log-uniform in [64 B, 256 MiB], dtype
                  uniform over {u8,i64,f16,bf16,f32}; recompute = exact copy,
                  a seeded 30 % with one random bit flipped
  [5] mass banks  2048 sessions, n ~ U[256,4096]; key bf16[512] ~ N(0,1);
                  value u8[2048] ~ U; query bf16[512]; host budget 8 GiB
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

SEED_BASE = 0x5EED0000

DTYPES_CLASSIFY = (torch.uint8, torch.int64, torch.float16, torch.bfloat16, torch.float32)


def seed_for(config_id: int) -> int:
    return SEED_BASE + config_id


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _randbytes(n: int, g: torch.Generator, device) -> torch.Tensor:
    return torch.randint(0, 256, (n,), generator=g, device=device, dtype=torch.uint8)


# --------------------------------------------------------------------------
# [1] Markovian session: uint8 observation + generator state
# --------------------------------------------------------------------------

@dataclass
class Markov:
    obs: torch.Tensor        # uint8 [3, H, W]
    rng: torch.Tensor        # int64 [2] carrying (seed, offset) as u64 bits


def markov(seed: int = seed_for(1), shape=(3, 256, 256), device="cpu") -> Markov:
    g = _gen(seed, device)
    obs = torch.randint(0, 256, shape, generator=g, device=device, dtype=torch.uint8)
    rng = _randbytes(16, g, device).view(torch.int64).clone()
    return Markov(obs=obs, rng=rng)


def excursion(m: Markov, seed: int) -> None:
    """Overwrite both buffers in place with unrelated random bytes."""
    g = _gen(seed, m.obs.device)
    m.obs.copy_(torch.randint(0, 256, m.obs.shape, generator=g, device=m.obs.device,
                              dtype=torch.uint8))
    m.rng.copy_(_randbytes(16, g, m.rng.device).view(torch.int64))


# --------------------------------------------------------------------------
# [2] / [5] Ragged memory banks, stored CSR: rows of all sessions back to back
# --------------------------------------------------------------------------

@dataclass
class Banks:
    n: list                  # entries per session (host ints)
    entry_off: list          # CSR offsets, len S+1 (host ints)
    keys: torch.Tensor       # [sum n, D]  fp16 or bf16
    values: torch.Tensor     # [sum n, ...] bf16 latent or uint8 bytes
    queries: torch.Tensor    # [S, D]
    key_dim: int
    value_bytes: int         # bytes of one value row

    @property
    def sessions(self) -> int:
        return len(self.n)


def banks(seed: int, sessions: int, n_lo: int, n_hi: int, key_dim: int,
          key_dtype: torch.dtype, value_shape: tuple, value_dtype: torch.dtype,
          device="cpu") -> Banks:
    gh = _gen(seed, "cpu")
    n = torch.randint(n_lo, n_hi + 1, (sessions,), generator=gh).tolist()
    off = [0]
    for x in n:
        off.append(off[-1] + x)
    total = off[-1]
    g = _gen(seed + 1, device)
    keys = torch.randn(total, key_dim, generator=g, device=device, dtype=torch.float32).to(key_dtype)
    queries = torch.randn(sessions, key_dim, generator=g, device=device,
                          dtype=torch.float32).to(key_dtype)
    if value_dtype == torch.uint8:
        values = torch.randint(0, 256, (total,) + tuple(value_shape), generator=g, device=device,
                               dtype=torch.uint8)
    else:
        values = torch.randn((total,) + tuple(value_shape), generator=g, device=device,
                             dtype=torch.float32).to(value_dtype)
    vb = values.element_size() * math.prod(value_shape)
    return Banks(n=n, entry_off=off, keys=keys, values=values, queries=queries,
                 key_dim=key_dim, value_bytes=vb)


def banks_config2(device="cpu", sessions=64, n_lo=1, n_hi=512, seed=seed_for(2)) -> Banks:
    return banks(seed, sessions, n_lo, n_hi, 256, torch.float16, (16, 32, 32), torch.bfloat16,
                 device)


def banks_config5(device="cpu", sessions=2048, n_lo=256, n_hi=4096, seed=seed_for(5)) -> Banks:
    return banks(seed, sessions, n_lo, n_hi, 512, torch.bfloat16, (2048,), torch.uint8, device)


# --------------------------------------------------------------------------
# [3] Windowed paged KV context
# --------------------------------------------------------------------------

@dataclass
class KV:
    k_pool: torch.Tensor     # bf16 [n_pages, page_rows, heads, head_dim]
    v_pool: torch.Tensor
    page_table: torch.Tensor # int32 [S, layers, window // page_rows]
    ring_start: list         # host ints, per session
    meta: torch.Tensor       # int64 [S, 4] position indices (global/local end, ...)
    layers: int
    window: int
    page_rows: int

    @property
    def sessions(self) -> int:
        return self.page_table.shape[0]

    @property
    def row_bytes(self) -> int:
        return self.k_pool[0, 0].numel() * self.k_pool.element_size()


def page_permutation(seed: int, sessions: int, layers: int, pages: int, device="cpu"):
    """A random assignment of every (session, layer, ring page) to a pool page."""
    g = _gen(seed, device)
    perm = torch.randperm(sessions * layers * pages, generator=g, device=device)
    return perm.to(torch.int32).view(sessions, layers, pages)


def kv(seed: int = seed_for(3), sessions=256, layers=24, heads=16, head_dim=64, window=1024,
       page_rows=16, device="cpu", fill=True) -> KV:
    assert window % page_rows == 0
    pages = window // page_rows
    n_pages = sessions * layers * pages
    gh = _gen(seed, "cpu")
    ring_start = torch.randint(0, window, (sessions,), generator=gh).tolist()
    meta = torch.randint(0, 2**40, (sessions, 4), generator=gh, dtype=torch.int64)
    page_table = page_permutation(seed + 1, sessions, layers, pages, device)
    shape = (n_pages, page_rows, heads, head_dim)
    k_pool = torch.empty(shape, device=device, dtype=torch.bfloat16)
    v_pool = torch.empty(shape, device=device, dtype=torch.bfloat16)
    if fill:
        g = _gen(seed + 2, device)
        # fill page by page block to bound the fp32 temporary
        step = max(1, (1 << 26) // (page_rows * heads * head_dim))
        for pool in (k_pool, v_pool):
            for p0 in range(0, n_pages, step):
                p1 = min(n_pages, p0 + step)
                pool[p0:p1].copy_(torch.randn((p1 - p0,) + shape[1:], generator=g, device=device,
                                              dtype=torch.float32))
    return KV(k_pool=k_pool, v_pool=v_pool, page_table=page_table, ring_start=ring_start,
              meta=meta.to(device), layers=layers, window=window, page_rows=page_rows)


# --------------------------------------------------------------------------
# [4] Classification sweep: buffers and a "recompute" pass
# --------------------------------------------------------------------------

@dataclass
class Sweep:
    before: list             # tensors (varied dtypes), as first computed
    after: list              # recompute pass: copies, some with one bit flipped
    flipped: list            # bool per buffer (ground truth of "changed")
    bit: list                # flipped bit position per buffer (-1 if none)
    sizes: list              # bytes per buffer


def sweep_sizes(seed: int, n: int, lo: int, hi: int):
    gh = _gen(seed, "cpu")
    u = torch.rand(n, generator=gh, dtype=torch.float64).tolist()
    dt = torch.randint(0, len(DTYPES_CLASSIFY), (n,), generator=gh).tolist()
    sizes, dtypes = [], []
    for ui, di in zip(u, dt):
        dtype = DTYPES_CLASSIFY[di]
        es = torch.tensor([], dtype=dtype).element_size()
        b = int(math.exp(math.log(lo) + ui * (math.log(hi) - math.log(lo))))
        b = max(es, b - b % es)
        sizes.append(b)
        dtypes.append(dtype)
    return sizes, dtypes


def sweep(seed: int = seed_for(4), n=200, lo=64, hi=1 << 28, frac=0.3, device="cpu",
          sizes=None, dtypes=None) -> Sweep:
    if sizes is None:
        sizes, dtypes = sweep_sizes(seed, n, lo, hi)
    n = len(sizes)
    gh = _gen(seed + 1, "cpu")
    n_flip = int(round(frac * n))
    chosen = set(torch.randperm(n, generator=gh)[:n_flip].tolist())
    g = _gen(seed + 2, device)
    before, after, flipped, bits = [], [], [], []
    for i, (b, dtype) in enumerate(zip(sizes, dtypes)):
        raw = _randbytes(b, g, device)
        t = raw.view(dtype)
        before.append(t)
        r2 = raw.clone()
        if i in chosen:
            bit = int(torch.randint(0, 8 * b, (1,), generator=gh).item())
            r2[bit // 8] ^= (1 << (bit % 8))
            bits.append(bit)
        else:
            bits.append(-1)
        after.append(r2.view(dtype))
        flipped.append(i in chosen)
    return Sweep(before=before, after=after, flipped=flipped, bit=bits, sizes=list(sizes))
