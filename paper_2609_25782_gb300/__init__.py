"""GB300-native hot path of the hot-cold KV hierarchy for agentic LLM serving.

Baek et al., "Hot-Cold Tiering of HBM and High Bandwidth Flash for Agentic LLM
Serving": active sessions' KV (the hot set) stays in HBM and is read by every
decode step; paused sessions' KV (the cold pool) lives in a second tier and
moves only on pause (pack) and resume (unpack). Here both tiers are device
memory of one GB300; the CUDA kernels and the pool runtime are in
``libkvtier.so`` (C ABI: include/kvtier.h), bound by :mod:`.kvtier`.

:class:`Pool` is a convenience owner: it allocates the two arenas with torch
(device memory only) and forwards every operation to the C ABI.
"""
from __future__ import annotations

from . import kvtier
from .kvtier import KVError  # noqa: F401

__all__ = ["Pool", "kvtier", "KVError"]


class Pool:
    def __init__(self, *, num_layers: int, num_hot_blocks: int, cold_bytes: int,
                 num_q_heads: int = 32, num_kv_heads: int = 4, head_dim: int = 128,
                 block_tokens: int = 16, max_sessions: int = 64, max_batch: int = 64,
                 max_context: int = 32768, alloc_seed: int = 0, device: int = 0,
                 lru_residency: bool = False):
        import torch
        self.device = torch.device("cuda", device)
        self.L, self.Hq, self.Hkv, self.D, self.bt = (num_layers, num_q_heads, num_kv_heads,
                                                      head_dim, block_tokens)
        self.num_hot_blocks = num_hot_blocks
        probe = kvtier.make_config(num_layers=num_layers, num_q_heads=num_q_heads,
                                   num_kv_heads=num_kv_heads, head_dim=head_dim,
                                   block_tokens=block_tokens, num_hot_blocks=num_hot_blocks)
        self.block_bytes = kvtier.kv_block_bytes(probe)
        self.token_bytes = kvtier.kv_token_bytes(probe)
        self.hot = torch.empty(num_hot_blocks * self.block_bytes // 2, dtype=torch.bfloat16,
                               device=self.device)
        self.cold = torch.empty(max(cold_bytes, 256) // 2, dtype=torch.bfloat16, device=self.device)
        cfg = kvtier.make_config(num_layers=num_layers, num_q_heads=num_q_heads,
                                 num_kv_heads=num_kv_heads, head_dim=head_dim,
                                 block_tokens=block_tokens, max_sessions=max_sessions,
                                 max_batch=max_batch, device=device, max_context=max_context,
                                 num_hot_blocks=num_hot_blocks, hot_base=self.hot,
                                 cold_bytes=cold_bytes, cold_base=self.cold, alloc_seed=alloc_seed,
                                 flags=kvtier.KV_POOL_LRU_RESIDENCY if lru_residency else 0)
        self.handle = kvtier.kv_pool_create(cfg)
        self.max_context = max_context

    def close(self) -> None:
        if getattr(self, "handle", None):
            kvtier.kv_pool_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # views -----------------------------------------------------------------
    def hot_view(self):
        """The hot arena as [NB][L][2][Hkv][bt][D] bf16."""
        return self.hot.view(self.num_hot_blocks, self.L, 2, self.Hkv, self.bt, self.D)

    def image(self, sid: int):
        """A session's cold image as [L][2][Hkv][T_cap][D] bf16 (a view)."""
        info = kvtier.session_info(self.handle, sid)
        off = (info.image - self.cold.data_ptr()) // 2
        n = self.L * 2 * self.Hkv * info.capacity * self.D
        return self.cold[off:off + n].view(self.L, 2, self.Hkv, info.capacity, self.D)

    # C ABI forwards ------------------------------------------------------------
    def session_create(self, max_tokens: int) -> int:
        return kvtier.session_create(self.handle, max_tokens)

    def session_create_paused(self, max_tokens: int, tokens: int) -> int:
        return kvtier.session_create_paused(self.handle, max_tokens, tokens)

    def session_destroy(self, sid: int) -> None:
        kvtier.session_destroy(self.handle, sid)

    def session_append(self, sid: int, k, v, stream=None) -> None:
        """k, v: device bf16 [L][n][Hkv][D]."""
        kvtier.session_append(self.handle, sid, k, v, int(k.shape[1]), stream)

    def session_pause(self, sid: int, stream=None) -> None:
        kvtier.session_pause(self.handle, sid, stream)

    def session_resume(self, sid: int, stream=None) -> None:
        kvtier.session_resume(self.handle, sid, stream)

    def session_info(self, sid: int):
        return kvtier.session_info(self.handle, sid)

    def session_block_table(self, sid: int) -> list[int]:
        return kvtier.session_block_table(self.handle, sid)

    def session_ready_event(self, sid: int):
        return kvtier.session_ready_event(self.handle, sid)

    def batch_tables(self, sids, block_tables, max_blocks: int, seq_lens, stream=None) -> None:
        kvtier.kv_pool_batch_tables(self.handle, list(sids), block_tables, max_blocks, seq_lens,
                                    stream)

    def batch_reserve(self, sids, block_tables, max_blocks: int, seq_lens, stream=None) -> None:
        """One new position per session (filled by decode_append_attention),
        then the batch's tables and lengths as batch_tables builds them."""
        kvtier.kv_pool_batch_reserve(self.handle, list(sids), block_tables, max_blocks, seq_lens,
                                     stream)

    def prefetch(self, next_sids, busy=(), stream=None) -> None:
        """Fetch the next step's evicted blocks ahead of it (residency mode),
        victims outside next_sids and busy (the step still being decoded)."""
        kvtier.kv_pool_prefetch(self.handle, list(next_sids), list(busy), stream)

    def session_block_table_device(self, sid: int) -> tuple[int, int]:
        """(device address of the session's table row, logical blocks)."""
        return kvtier.session_block_table_device(self.handle, sid)

    def decode_attention(self, layer: int, q, block_tables, seq_lens, B: int, max_blocks: int,
                         scale: float, out, stream=None, overlap_previous: bool = False) -> None:
        """out: fp32, or bf16 (then the result is rounded to nearest even)."""
        import torch
        flags = (kvtier.KV_DECODE_OVERLAP_PREVIOUS if overlap_previous else 0) | \
            (kvtier.KV_DECODE_OUT_BF16 if getattr(out, "dtype", None) == torch.bfloat16 else 0)
        if flags:
            kvtier.decode_attention_ex(self.handle, layer, q, block_tables, seq_lens, B,
                                       max_blocks, scale, out, flags, stream)
        else:
            kvtier.decode_attention(self.handle, layer, q, block_tables, seq_lens, B, max_blocks,
                                    scale, out, stream)

    def decode_append_attention(self, layer: int, q, k_new, v_new, block_tables, seq_lens, B: int,
                                max_blocks: int, scale: float, out, stream=None,
                                overlap_previous: bool = False) -> None:
        """k_new, v_new: device bf16 [B][Hkv][D] (leading [L] for layer -1), the
        token at seq_lens[b] - 1 of each row, written to the pool and attended to."""
        import torch
        flags = (kvtier.KV_DECODE_OVERLAP_PREVIOUS if overlap_previous else 0) | \
            (kvtier.KV_DECODE_OUT_BF16 if getattr(out, "dtype", None) == torch.bfloat16 else 0)
        kvtier.decode_append_attention(self.handle, layer, q, k_new, v_new, block_tables, seq_lens,
                                       B, max_blocks, scale, out, flags, stream)

    def shuffle_free(self, seed: int) -> None:
        kvtier.kv_pool_shuffle_free(self.handle, seed)

    def free_list(self) -> list[int]:
        return kvtier.kv_pool_free_list(self.handle)

    def stats(self) -> dict:
        return kvtier.kv_pool_get_stats(self.handle)

    def check_device(self) -> int:
        return kvtier.kv_pool_check_device(self.handle)
