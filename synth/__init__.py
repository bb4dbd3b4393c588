"""Seeded synthetic inputs for the hot/cold KV path.

This module draws inputs only: session lengths, physical block placements, and
the bf16 values of queries, keys and values. It holds none of the attention or
migration arithmetic, and it is the one module that both the CPU oracle side
and the CUDA side of the tests and benchmarks import.

Values are produced by a counter-based generator so that any element can be
regenerated on its own, on the host (numpy) or on the device (torch integer
ops), bit for bit:

* ``hash64(key, i)`` is the splitmix64 output function (Steele, Lea and Flood,
  "Fast splittable pseudorandom number generators", OOPSLA 2014; constants as
  in Vigna's public-domain splitmix64.c) applied to ``key + (i + 1) * GAMMA``.
* A 64-bit hash is cut into four 16-bit uniforms whose sum, centred and scaled
  to unit variance, is an Irwin-Hall(4) approximation of N(0, 1) (support
  +-3.46 sigma, excess kurtosis -0.3). The integer sum is exact in fp32, the
  scale is one fp32 multiply, and the bf16 conversion is round-to-nearest-even,
  so both sides produce identical bits.

Logical coordinates of a K/V element are (session id, layer, kv, kv-head,
token, dim); the element's counter packs them into 57 bits (token < 2**20,
layer < 64, kv-head < 8, dim < 128, session id < 2**20).
"""
from __future__ import annotations

import math

import numpy as np

M64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB
KEYMUL = 0xD1B54A32D192ED03

SALT_KV = 0x4B56
SALT_Q = 0x5131

# 1 / std of the sum of four independent uniforms on {0..65535}
_IH_CENTER = 4 * 65535 // 2          # 131070
_IH_SCALE = np.float32(1.0 / math.sqrt((65536.0 ** 2 - 1.0) / 3.0))

BF16_NAN = 0x7FC0


def _u64(x: int) -> np.uint64:
    return np.uint64(x & M64)


def key_of(seed: int, salt: int) -> int:
    """64-bit stream key for (seed, salt): splitmix64 finaliser of a mix."""
    z = (seed * KEYMUL + salt * GAMMA + 1) & M64
    z = ((z ^ (z >> 30)) * MIX1) & M64
    z = ((z ^ (z >> 27)) * MIX2) & M64
    return z ^ (z >> 31)


# --------------------------------------------------------------------------
# numpy (host) side
# --------------------------------------------------------------------------

def hash64_np(key: int, idx: np.ndarray) -> np.ndarray:
    idx = np.asarray(idx, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = _u64(key) + (idx + np.uint64(1)) * _u64(GAMMA)
        z = (z ^ (z >> np.uint64(30))) * _u64(MIX1)
        z = (z ^ (z >> np.uint64(27))) * _u64(MIX2)
        z = z ^ (z >> np.uint64(31))
    return z


def f32_to_bf16_bits_np(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16 bit patterns (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    with np.errstate(over="ignore"):
        return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32_np(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_bf16_np(key: int, idx: np.ndarray, scale: float = 1.0) -> np.ndarray:
    """bf16 bits of an approximately N(0, 1) value (times ``scale``)."""
    h = hash64_np(key, idx)
    m = np.uint64(0xFFFF)
    s = (h & m) + ((h >> np.uint64(16)) & m) + ((h >> np.uint64(32)) & m) + (h >> np.uint64(48))
    z = (s.astype(np.int64) - _IH_CENTER).astype(np.float32) * _IH_SCALE
    if scale != 1.0:
        z = z * np.float32(scale)
    return f32_to_bf16_bits_np(z)


def kv_index_np(sess, layer, kv, g, t, d):
    """Counter of a K/V element; arguments broadcast like numpy arrays."""
    sess = np.asarray(sess, dtype=np.uint64)
    base = ((sess * np.uint64(64) + np.asarray(layer, dtype=np.uint64)) * np.uint64(2)
            + np.asarray(kv, dtype=np.uint64)) * np.uint64(8) + np.asarray(g, dtype=np.uint64)
    return (base << np.uint64(27)) | (np.asarray(t, dtype=np.uint64) << np.uint64(7)) \
        | np.asarray(d, dtype=np.uint64)


def q_index_np(sess, layer, h, d):
    sess = np.asarray(sess, dtype=np.uint64)
    base = (sess * np.uint64(64) + np.asarray(layer, dtype=np.uint64)) * np.uint64(64) \
        + np.asarray(h, dtype=np.uint64)
    return (base << np.uint64(7)) | np.asarray(d, dtype=np.uint64)


def session_kv_np(seed: int, sess: int, layers, num_kv_heads: int, head_dim: int,
                  tokens: int, k_scale: float = 1.0):
    """Logical K and V of one session: two uint16 arrays [len(layers)][Hkv][T][D]."""
    key = key_of(seed, SALT_KV)
    layers = np.asarray(list(layers), dtype=np.uint64)
    l = layers[:, None, None, None]
    g = np.arange(num_kv_heads, dtype=np.uint64)[None, :, None, None]
    t = np.arange(tokens, dtype=np.uint64)[None, None, :, None]
    d = np.arange(head_dim, dtype=np.uint64)[None, None, None, :]
    k = normal_bf16_np(key, kv_index_np(sess, l, 0, g, t, d), k_scale)
    v = normal_bf16_np(key, kv_index_np(sess, l, 1, g, t, d), 1.0)
    return k, v


def token_kv_np(seed: int, sess: int, layer: int, t: int, num_kv_heads: int, head_dim: int,
                k_scale: float = 1.0):
    """K and V of one token of one layer: two uint16 arrays [Hkv][D]."""
    key = key_of(seed, SALT_KV)
    g = np.arange(num_kv_heads, dtype=np.uint64)[:, None]
    d = np.arange(head_dim, dtype=np.uint64)[None, :]
    k = normal_bf16_np(key, kv_index_np(sess, layer, 0, g, t, d), k_scale)
    v = normal_bf16_np(key, kv_index_np(sess, layer, 1, g, t, d), 1.0)
    return k, v


def queries_np(seed: int, sess_ids, layers, num_q_heads: int, head_dim: int):
    """Q bits [len(layers)][len(sess_ids)][Hq][D] uint16."""
    key = key_of(seed, SALT_Q)
    s = np.asarray(list(sess_ids), dtype=np.uint64)[None, :, None, None]
    l = np.asarray(list(layers), dtype=np.uint64)[:, None, None, None]
    h = np.arange(num_q_heads, dtype=np.uint64)[None, None, :, None]
    d = np.arange(head_dim, dtype=np.uint64)[None, None, None, :]
    return normal_bf16_np(key, q_index_np(s, l, h, d))


def session_lengths(seed: int, n: int, lo: int, hi: int, block_tokens: int = 16,
                    need_partial: bool = True) -> np.ndarray:
    """n integer lengths uniform on [lo, hi]; with need_partial, at least one
    length is not a multiple of block_tokens when [lo, hi] holds one."""
    rng = np.random.Generator(np.random.PCG64(seed))
    t = rng.integers(lo, hi + 1, size=n).astype(np.int64)
    if need_partial and n > 0 and np.all(t % block_tokens == 0):
        if t[0] - 1 >= lo:
            t[0] -= 1
        elif t[0] + 1 <= hi:
            t[0] += 1
    return t


def random_block_tables(seed: int, seq_lens, block_tokens: int, num_blocks: int,
                        max_blocks: int | None = None) -> np.ndarray:
    """Block tables [B][max_blocks] int32 drawing distinct physical blocks from
    a seeded random permutation of range(num_blocks); unused entries are -1."""
    seq_lens = np.asarray(seq_lens, dtype=np.int64)
    need = -(-seq_lens // block_tokens)
    if max_blocks is None:
        max_blocks = int(need.max()) if len(need) else 1
    if int(need.sum()) > num_blocks:
        raise ValueError("pool too small for the requested sessions")
    rng = np.random.Generator(np.random.PCG64(seed ^ 0x7AB1E))
    perm = rng.permutation(num_blocks).astype(np.int32)
    tables = np.full((len(seq_lens), max_blocks), -1, dtype=np.int32)
    pos = 0
    for b, n in enumerate(need):
        tables[b, :n] = perm[pos:pos + n]
        pos += int(n)
    return tables


def hot_pool_np(seed: int, sess_ids, seq_lens, tables, num_blocks: int, layers: int,
                num_kv_heads: int, head_dim: int, block_tokens: int, k_scale: float = 1.0,
                poison_tail: bool = True) -> np.ndarray:
    """Host hot pool [NB][L][2][Hkv][bt][D] (uint16 bf16 bits) holding each
    session's logical K/V in the physical blocks named by its table row.
    Unused slots hold bf16 NaN when poison_tail is set (zeros otherwise)."""
    fill = BF16_NAN if poison_tail else 0
    hot = np.full((num_blocks, layers, 2, num_kv_heads, block_tokens, head_dim), fill,
                  dtype=np.uint16)
    for b, (sid, T) in enumerate(zip(sess_ids, seq_lens)):
        T = int(T)
        k, v = session_kv_np(seed, int(sid), range(layers), num_kv_heads, head_dim, T, k_scale)
        nblk = -(-T // block_tokens)
        for j in range(nblk):
            p = int(tables[b][j])
            t0, t1 = j * block_tokens, min(T, (j + 1) * block_tokens)
            hot[p, :, 0, :, : t1 - t0, :] = k[:, :, t0:t1, :]
            hot[p, :, 1, :, : t1 - t0, :] = v[:, :, t0:t1, :]
    return hot


def session_image_np(seed: int, sess: int, layers: int, num_kv_heads: int, head_dim: int,
                     tokens: int, cap: int, k_scale: float = 1.0,
                     poison_tail: bool = True) -> np.ndarray:
    """Host cold image [L][2][Hkv][cap][D] of one session (first ``tokens`` valid)."""
    img = np.full((layers, 2, num_kv_heads, cap, head_dim), BF16_NAN if poison_tail else 0,
                  dtype=np.uint16)
    k, v = session_kv_np(seed, sess, range(layers), num_kv_heads, head_dim, tokens, k_scale)
    img[:, 0, :, :tokens, :] = k
    img[:, 1, :, :tokens, :] = v
    return img


# --------------------------------------------------------------------------
# torch (device) side: the same integer recipe, for inputs too large to
# generate on the host. Imported lazily so the numpy side needs no torch.
# --------------------------------------------------------------------------

def _s64(x: int) -> int:
    x &= M64
    return x - (1 << 64) if x >= (1 << 63) else x


def _lsr(x, k: int):
    return (x >> k) & ((1 << (64 - k)) - 1)


def hash64_torch(key: int, idx):
    z = idx + 1
    z = z * _s64(GAMMA) + _s64(key)
    z = (z ^ _lsr(z, 30)) * _s64(MIX1)
    z = (z ^ _lsr(z, 27)) * _s64(MIX2)
    return z ^ _lsr(z, 31)


def normal_bf16_torch(key: int, idx, scale: float = 1.0):
    """Same bits as normal_bf16_np, as a torch.bfloat16 tensor."""
    import torch
    h = hash64_torch(key, idx)
    s = (h & 0xFFFF) + (_lsr(h, 16) & 0xFFFF) + (_lsr(h, 32) & 0xFFFF) + _lsr(h, 48)
    z = (s - _IH_CENTER).to(torch.float32) * float(_IH_SCALE)
    if scale != 1.0:
        z = z * float(np.float32(scale))
    return z.to(torch.bfloat16)


def _kv_index_torch(sess, layer, kv, g, t, d):
    base = ((sess * 64 + layer) * 2 + kv) * 8 + g
    return (base << 27) | (t << 7) | d


def fill_hot_pool_torch(hot, seed: int, sess_ids, seq_lens, tables, layers: int,
                        num_kv_heads: int, head_dim: int, block_tokens: int,
                        k_scale: float = 1.0, poison_tail: bool = True,
                        chunk_blocks: int = 32):
    """Write each session's logical K/V into ``hot`` (torch bf16 tensor viewed
    as [NB][L][2][Hkv][bt][D]) at the physical blocks of its table row, with
    torch ops on hot's device. Same values as hot_pool_np."""
    import torch
    dev = hot.device
    key = key_of(seed, SALT_KV)
    L, H, D, bt = layers, num_kv_heads, head_dim, block_tokens
    l = torch.arange(L, device=dev, dtype=torch.int64).view(1, L, 1, 1, 1, 1)
    kv = torch.arange(2, device=dev, dtype=torch.int64).view(1, 1, 2, 1, 1, 1)
    g = torch.arange(H, device=dev, dtype=torch.int64).view(1, 1, 1, H, 1, 1)
    s = torch.arange(bt, device=dev, dtype=torch.int64).view(1, 1, 1, 1, bt, 1)
    d = torch.arange(D, device=dev, dtype=torch.int64).view(1, 1, 1, 1, 1, D)
    scale_k = torch.ones(1, 1, 2, 1, 1, 1, device=dev, dtype=torch.float32)
    if k_scale != 1.0:
        scale_k[:, :, 0] = float(np.float32(k_scale))
    hv = hot.view(-1, L, 2, H, bt, D)
    nan = torch.tensor(float("nan"), dtype=torch.bfloat16, device=dev)
    for b, (sid, T) in enumerate(zip(sess_ids, seq_lens)):
        T = int(T)
        nblk = -(-T // bt)
        row = torch.as_tensor(np.asarray(tables[b][:nblk], dtype=np.int64), device=dev)
        for j0 in range(0, nblk, chunk_blocks):
            j1 = min(nblk, j0 + chunk_blocks)
            j = torch.arange(j0, j1, device=dev, dtype=torch.int64).view(-1, 1, 1, 1, 1, 1)
            t = j * bt + s
            idx = _kv_index_torch(int(sid), l, kv, g, t, d)
            hsh = hash64_torch(key, idx)
            sm = (hsh & 0xFFFF) + (_lsr(hsh, 16) & 0xFFFF) + (_lsr(hsh, 32) & 0xFFFF) + _lsr(hsh, 48)
            z = (sm - _IH_CENTER).to(torch.float32) * float(_IH_SCALE)
            if k_scale != 1.0:
                z = z * scale_k
            vals = z.to(torch.bfloat16)
            if poison_tail and j1 * bt > T:
                vals = torch.where(t.expand_as(vals) < T, vals, nan)
            hv[row[j0:j1]] = vals
    return hot


def fill_image_torch(img, seed: int, sess: int, layers: int, num_kv_heads: int,
                     head_dim: int, tokens: int, k_scale: float = 1.0,
                     chunk_tokens: int = 4096):
    """Write one session's logical K/V into a torch bf16 image [L][2][Hkv][cap][D]."""
    import torch
    dev = img.device
    key = key_of(seed, SALT_KV)
    L, H, D = layers, num_kv_heads, head_dim
    iv = img.view(L, 2, H, -1, D)
    l = torch.arange(L, device=dev, dtype=torch.int64).view(L, 1, 1, 1, 1)
    kv = torch.arange(2, device=dev, dtype=torch.int64).view(1, 2, 1, 1, 1)
    g = torch.arange(H, device=dev, dtype=torch.int64).view(1, 1, H, 1, 1)
    d = torch.arange(D, device=dev, dtype=torch.int64).view(1, 1, 1, 1, D)
    scale_k = torch.ones(1, 2, 1, 1, 1, device=dev, dtype=torch.float32)
    scale_k[:, 0] = float(np.float32(k_scale))
    for t0 in range(0, tokens, chunk_tokens):
        t1 = min(tokens, t0 + chunk_tokens)
        t = torch.arange(t0, t1, device=dev, dtype=torch.int64).view(1, 1, 1, -1, 1)
        idx = _kv_index_torch(int(sess), l, kv, g, t, d)
        hsh = hash64_torch(key, idx)
        sm = (hsh & 0xFFFF) + (_lsr(hsh, 16) & 0xFFFF) + (_lsr(hsh, 32) & 0xFFFF) + _lsr(hsh, 48)
        z = (sm - _IH_CENTER).to(torch.float32) * float(_IH_SCALE)
        if k_scale != 1.0:
            z = z * scale_k
        iv[:, :, :, t0:t1, :] = z.to(torch.bfloat16)
    return img


def queries_torch(seed: int, sess_ids, layers, num_q_heads: int, head_dim: int, device):
    """Same bits as queries_np, as a torch bf16 tensor [L][B][Hq][D] on device."""
    import torch
    key = key_of(seed, SALT_Q)
    s = torch.as_tensor(np.asarray(list(sess_ids), dtype=np.int64), device=device).view(1, -1, 1, 1)
    l = torch.as_tensor(np.asarray(list(layers), dtype=np.int64), device=device).view(-1, 1, 1, 1)
    h = torch.arange(num_q_heads, device=device, dtype=torch.int64).view(1, 1, -1, 1)
    d = torch.arange(head_dim, device=device, dtype=torch.int64).view(1, 1, 1, -1)
    idx = (((s * 64 + l) * 64 + h) << 7) | d
    return normal_bf16_torch(key, idx)


def kv_logical_torch(seed: int, sess: int, layers, num_kv_heads: int, head_dim: int,
                     t0: int, t1: int, device, k_scale: float = 1.0):
    """Logical K and V rows [len(layers)][Hkv][t1-t0][D] as torch bf16 on device
    (used to build appended tokens)."""
    import torch
    key = key_of(seed, SALT_KV)
    l = torch.as_tensor(np.asarray(list(layers), dtype=np.int64), device=device).view(-1, 1, 1, 1)
    g = torch.arange(num_kv_heads, device=device, dtype=torch.int64).view(1, -1, 1, 1)
    t = torch.arange(t0, t1, device=device, dtype=torch.int64).view(1, 1, -1, 1)
    d = torch.arange(head_dim, device=device, dtype=torch.int64).view(1, 1, 1, -1)
    k = normal_bf16_torch(key, _kv_index_torch(int(sess), l, 0, g, t, d), k_scale)
    v = normal_bf16_torch(key, _kv_index_torch(int(sess), l, 1, g, t, d), 1.0)
    return k, v
