/*
 * kvtier.h - C ABI of the hot/cold KV tiering hot path for one GB300 GPU.
 *
 * The library implements the data paths of the hot-cold KV hierarchy of
 * Baek et al., "Hot-Cold Tiering of HBM and High Bandwidth Flash for Agentic
 * LLM Serving" (Section 3, "Architecture and data paths"):
 *   path 1  decode attention over the HBM-resident hot set ... decode_attention
 *   path 2  resume: cold image -> hot blocks ................ session_resume
 *   path 3  fresh KV written into hot blocks ................ session_append
 *           (or kv_pool_batch_reserve + decode_append_attention: one
 *           token per session and step, written by the decode kernel)
 *   path 4  eviction: hot blocks -> cold image .............. session_pause
 * The cold tier (high bandwidth flash in the paper) is a second device
 * allocation; its bandwidth, energy and endurance are not modelled.
 *
 * Data layout (all bf16, D = head_dim = 128, bt = block_tokens):
 *   hot pool   hot[num_hot_blocks][L][2][Hkv][bt][D]   (2 = K, V)
 *              One block holds bt tokens of every layer: 16 tokens x 96 KiB
 *              = 1.5 MiB for L=48, Hkv=4 (the paper's block unit, Section 4).
 *              Each (block, layer, K|V, kv-head) run is bt*D*2 = 4 KiB.
 *   cold image img[L][2][Hkv][T_cap][D] per session, contiguous and
 *              layer-major, placed in the cold arena by the pool.
 *   block table: row of int32 physical block ids; logical block j of a
 *              session holds its tokens j*bt .. j*bt+bt-1.
 *
 * Conventions for every call:
 *  - Return value 0 (KV_OK) or a negative KV_ERR_* code. On error nothing
 *    changes: no host state, no block ownership, no device work enqueued
 *    that would alter data. kv_last_error() describes the last failure of
 *    the calling thread.
 *  - Pointers documented as "device" are CUDA device addresses on the pool's
 *    device; "host" pointers are ordinary CPU memory read or written before
 *    the call returns.
 *  - Device work is enqueued on the given stream and is asynchronous; host
 *    metadata (states, lengths, tables, the free list) changes when the call
 *    returns. Streams are cudaStream_t values (kv_stream_t is the same type);
 *    0 is the legacy default stream.
 *  - The caller owns the hot and cold arenas, Q, outputs, batch tables and
 *    streams. The pool owns its metadata, a device block-table arena, the
 *    decode workspace and its CUDA events.
 *  - A pool is not thread-safe: one host thread at a time.
 */
#ifndef KVTIER_H
#define KVTIER_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *kv_stream_t; /* == cudaStream_t */
typedef struct CUevent_st *kv_event_t;   /* == cudaEvent_t  */
typedef struct kv_pool kv_pool;          /* opaque */

enum {
    KV_OK = 0,
    KV_ERR_INVALID_ARG = -1,   /* bad size, pointer, id or shape */
    KV_ERR_BAD_STATE = -2,     /* e.g. resume of an active session */
    KV_ERR_NO_HOT_BLOCKS = -3, /* free list cannot cover the request */
    KV_ERR_NO_COLD_SPACE = -4, /* cold arena cannot hold the image */
    KV_ERR_CUDA = -5,          /* a CUDA runtime call failed */
    KV_ERR_DEVICE_CHECK = -6   /* a kernel's own bounds check fired */
};

enum { KV_SESSION_FREE = 0, KV_SESSION_ACTIVE = 1, KV_SESSION_PAUSED = 2 };

/* Pool flag: bookkeeping only. No CUDA call is made, no kernel runs and no
 * data moves; calls that would compute return KV_ERR_BAD_STATE. Used to test
 * the host logic (placement, states, errors) on machines without a GPU. */
#define KV_POOL_HOST_LOGIC_ONLY 1u

/* Pool flag: block residency with LRU eviction (Section 3, "Eviction, resume
 * and decode"; Section 4: each 1.5 MiB block is resident in HBM, the cold
 * tier, or both, with write-back LRU). In this mode
 *  - session_pause moves nothing: a paused session's blocks stay hot and age;
 *  - when an allocation finds no free block, the least recently used hot
 *    blocks are evicted (sessions ordered by last use, i.e. the last append,
 *    resume or kv_pool_batch_tables that named them; ties by session id;
 *    within a session, ascending block index). Active blocks are not pinned;
 *    the sessions the current call works on are never its victims;
 *  - an evicted block is written to the session's image only for the tokens
 *    the image does not hold yet, so every token is written at most once
 *    (write-on-evict, Section 3, "Memory hierarchy and write policy");
 *  - session_resume fetches only the blocks that are no longer hot (the
 *    others count as resume hits), and kv_pool_batch_tables first fetches
 *    any evicted block of its sessions (kv_pool_prefetch fetches them one
 *    step ahead); a fetch waits for the evictions that wrote the session's
 *    image, whatever stream they ran on;
 *  - evicted slots go to the end of the free list, in eviction order, and the
 *    call's allocations pop from the end.
 * Any call that allocates may evict blocks of any other session, so order it
 * after the decode work that still reads the pool (evictions wait for the
 * victims' own appends and resumes by themselves). */
#define KV_POOL_LRU_RESIDENCY 2u

typedef struct kv_pool_config {
    int32_t num_layers;     /* L  (48 for Qwen3-Coder-30B-A3B)             */
    int32_t num_q_heads;    /* Hq (32); Hq / Hkv must be 1, 2, 4 or 8      */
    int32_t num_kv_heads;   /* Hkv (4), at most 8                          */
    int32_t head_dim;       /* D; must be 128                              */
    int32_t block_tokens;   /* bt; 16 or 64                                */
    int32_t max_sessions;   /* session ids are 0 .. max_sessions-1          */
    int32_t max_batch;      /* sizes the decode workspace (see decode_attention) */
    int32_t device;         /* CUDA ordinal holding both arenas             */
    int64_t max_context;    /* longest session in tokens (table width)      */
    int64_t num_hot_blocks; /* blocks in the hot arena                      */
    void *hot_base;         /* device, >= num_hot_blocks * block bytes, 256-B aligned */
    int64_t cold_bytes;     /* bytes in the cold arena                      */
    void *cold_base;        /* device, 256-B aligned                        */
    uint64_t alloc_seed;    /* seeds the shuffle of the initial free list   */
    uint32_t flags;         /* KV_POOL_HOST_LOGIC_ONLY | KV_POOL_LRU_RESIDENCY */
    uint32_t reserved;
} kv_pool_config;

typedef struct kv_session_info {
    int32_t state;       /* KV_SESSION_*                                   */
    int32_t num_blocks;  /* hot blocks held (simple mode: 0 when paused)   */
    int64_t tokens;      /* T: tokens in the session's KV                  */
    int64_t capacity;    /* T_cap of its cold image                        */
    int64_t cold_valid;  /* tokens already valid in the cold image         */
    void *image;         /* device address of img[L][2][Hkv][T_cap][D]     */
} kv_session_info;

typedef struct kv_pool_stats {
    int64_t free_blocks;
    int64_t used_blocks;
    int64_t cold_bytes_used;
    int64_t bytes_unpacked;   /* image bytes copied cold -> hot (path 2)   */
    int64_t bytes_packed;     /* image bytes copied hot -> cold (path 4)   */
    int64_t bytes_appended;   /* KV bytes of tokens added by session_append
                               * and kv_pool_batch_reserve                  */
    int64_t resumes, pauses, appends, decodes; /* appends: calls, plus one per
                                                * reserved batch member    */
    int64_t blocks_evicted;       /* residency mode: blocks evicted            */
    int64_t resume_blocks_hit;    /* residency mode: still hot at resume       */
    int64_t resume_blocks_missed; /* residency mode: fetched at resume         */
    int64_t batch_blocks_fetched; /* residency mode: fetched by kv_pool_batch_tables
                                   * or kv_pool_batch_reserve (inside a step)  */
    int64_t blocks_prefetched;    /* residency mode: fetched by kv_pool_prefetch */
    int64_t prefetches;           /* kv_pool_prefetch calls that did their work */
} kv_pool_stats;

/* Create a pool over caller-owned arenas. Bookkeeping; no passage of the
 * paper defines pool set-up. What it sets up does have one: the hot pool of
 * fixed-size paged blocks (Section 2, "Large Language Models"; one block =
 * 16 tokens of every layer, the 1.5 MiB unit of Section 4, "Methodology")
 * and the cold pool of per-session images (Section 3, "Architecture and
 * data paths"). The hot free list starts as 0..num_hot_blocks-1 shuffled by
 * Fisher-Yates driven by splitmix64 seeded with alloc_seed (draw
 * j = floor(r * (i+1) / 2^64) for i = n-1 .. 1); allocations pop from its
 * end. Allocates the pool's device metadata (tables, decode workspace, flag
 * word) with cudaMalloc. *out receives the pool. Errors: bad shape or null
 * or misaligned arenas -> KV_ERR_INVALID_ARG; a failing CUDA call ->
 * KV_ERR_CUDA (nothing is left allocated). */
int kv_pool_create(const kv_pool_config *cfg, kv_pool **out);

/* Destroy a pool after synchronising its device. Bookkeeping; no passage.
 * Frees the pool's own device metadata and events; the caller's arenas are
 * not freed. */
int kv_pool_destroy(kv_pool *pool);

/* Bytes of one hot block: L * 2 * Hkv * bt * D * 2. */
int64_t kv_block_bytes(const kv_pool_config *cfg);

/* Bytes of K plus V per token: L * 2 * Hkv * D * 2 (96 KiB for the paper's
 * model, Section 4). */
int64_t kv_token_bytes(const kv_pool_config *cfg);

/* S(t): the most KV splits a decode call makes for one (session, head) of up
 * to t tokens, the factor by which the decode workspace scales (see
 * decode_attention). Each session of T tokens is cut into ceil(T/16) 16-token
 * tiles and split every clamp(ceil(tiles/16), 64, 128) tiles, a function of T
 * alone. Returns 0 for t < 1. */
int32_t kv_decode_splits(int64_t t);

/* Create an ACTIVE, empty session able to hold max_tokens (1 ..
 * max_context) tokens. Bookkeeping; no passage defines the call. A session
 * is the paper's unit of agentic serving, whose context keeps growing
 * across turns (Section 2, "Agentic AI Serving"); its cold image is the
 * per-session region that data path 4 writes (Section 3). Reserves the
 * image (max_tokens * token bytes, rounded up to 256 B) in the cold arena
 * (first fit). Errors: KV_ERR_NO_COLD_SPACE, too many sessions ->
 * KV_ERR_INVALID_ARG. */
int session_create(kv_pool *pool, int64_t max_tokens, int32_t *sid_out);

/* Create a PAUSED session whose image the caller fills with `tokens` valid
 * tokens (session_info gives its device address); cold_valid = tokens. */
int session_create_paused(kv_pool *pool, int64_t max_tokens, int64_t tokens,
                          int32_t *sid_out);

/* Release a session's hot blocks and cold image (any state). The caller
 * must have finished all work that reads them. */
int session_destroy(kv_pool *pool, int32_t sid);

/* Data path 3 (Section 3): write n >= 1 new tokens of an ACTIVE session.
 * k, v: device, bf16 [L][n][Hkv][D] contiguous, 16-byte aligned. Blocks are popped from the
 * free list when the tail block fills; tokens go to positions T .. T+n-1,
 * then T += n. The stream first waits for the session's last resume.
 * Errors: KV_ERR_BAD_STATE (paused), KV_ERR_NO_HOT_BLOCKS, capacity
 * exceeded -> KV_ERR_INVALID_ARG. */
int session_append(kv_pool *pool, int32_t sid, const void *k, const void *v, int32_t n,
                   kv_stream_t stream);

/* Data path 1 (Section 3; Section 2: decoding attends to the cached KV):
 * one decode step of grouped-query attention for B sessions.
 *   layer        0 .. L-1, or -1 for all layers in one launch (q and out
 *                then carry a leading [L] dimension)
 *   q            device bf16 [B][Hq][D]   (or [L][B][Hq][D])
 *   block_tables device int32 [B][max_blocks]; row b lists session b's
 *                blocks in logical order. max_blocks sizes the grid (splits
 *                for max_blocks * bt tokens): the batch's longest session is
 *                the best width
 *   seq_lens     device int32 [B]; 1 <= seq_lens[b] <= max_blocks * bt
 *   scale        multiplies q.k before the softmax (1/sqrt(D) usually)
 *   out          device fp32 [B][Hq][D]   (or [L][B][Hq][D]), 16-byte aligned
 *                (q, block_tables and seq_lens 4-byte aligned; misaligned
 *                pointers -> KV_ERR_INVALID_ARG)
 * out[b][h] = sum_i softmax_i(scale * q[b][h] . K[g][i]) V[g][i] over the
 * session's tokens i < seq_lens[b], g = h / (Hq/Hkv). Tokens past seq_len
 * in the last block are never read into the result (they may hold NaN).
 * The result depends only on the values and seq_lens: not on physical
 * placement, batch composition or timing (bit-identical across a
 * pause/resume round trip). The pool's decode workspace holds
 * max_batch x Hq x S(max_context) partial rows, S(t) = kv_decode_splits(t)
 * (ceil(t / 1024) up to 16 splits, ceil(t / 2048) beyond 32K tokens); a
 * call needs
 * layers x B x Hq x S(max_blocks x bt) rows, else KV_ERR_INVALID_ARG. Calls on
 * one pool share the workspace (the partials, and one split-arrival counter
 * per (row, kv-head) that every call leaves at zero): issue them in order on
 * one stream. Calls whose work overlaps on the GPU give wrong results, and
 * counters they leave non-zero make later multi-split results wrong too. */
int decode_attention(kv_pool *pool, int32_t layer, const void *q,
                     const int32_t *block_tables, const int32_t *seq_lens, int32_t B,
                     int32_t max_blocks, float scale, float *out, kv_stream_t stream);

/* decode_attention with options. KV_DECODE_OVERLAP_PREVIOUS lets this
 * call's split kernel start while the kernel just before it on the stream is
 * still running (programmatic dependent launch): it reads block ids and
 * prefetches K/V tiles at once, and waits for that kernel to finish before
 * it reads q (or k_new, v_new) or writes out, the workspace or the pool. The
 * caller promises that the kernel just before it on the stream (typically
 * the previous layer's decode call) writes neither block_tables, seq_lens
 * nor any hot-arena row of the layers this call reads; a
 * decode_append_attention call for another layer writes only its own
 * layer's rows and qualifies. flags = 0 is decode_attention. */
#define KV_DECODE_OVERLAP_PREVIOUS 1u
/* KV_DECODE_OUT_BF16: `out` is bf16 [..][Hq][D] (the fp32 result rounded to
 * nearest even), halving the output bytes for a caller that consumes bf16. */
#define KV_DECODE_OUT_BF16 2u
int decode_attention_ex(kv_pool *pool, int32_t layer, const void *q,
                        const int32_t *block_tables, const int32_t *seq_lens, int32_t B,
                        int32_t max_blocks, float scale, float *out, uint32_t flags,
                        kv_stream_t stream);

/* Data paths 3 and 1 fused (Section 3: the step's fresh KV is written into
 * HBM and decode reads it): decode_attention_ex where the newest token of
 * every batch row, position seq_lens[b] - 1, arrives with the call.
 *   k_new, v_new  device bf16 [B][Hkv][D] (or [L][B][Hkv][D] for layer =
 *                 -1), 16-byte aligned: that token's K and V
 * The kernel stores them into the token's pool slot, which
 * kv_pool_batch_reserve allocated (block_tables and seq_lens are its
 * outputs), and attends over tokens 0 .. seq_lens[b] - 1 including it.
 * Result and pool contents are bit-identical to session_append of the token
 * followed by decode_attention_ex. Issue it for every layer (or once with
 * layer = -1) before any call that may pack the sessions' blocks. Errors as
 * decode_attention_ex; null or misaligned k_new/v_new -> KV_ERR_INVALID_ARG. */
int decode_append_attention(kv_pool *pool, int32_t layer, const void *q, const void *k_new,
                            const void *v_new, const int32_t *block_tables,
                            const int32_t *seq_lens, int32_t B, int32_t max_blocks, float scale,
                            float *out, uint32_t flags, kv_stream_t stream);

/* Data path 4 with write-on-evict (Section 3, "Memory hierarchy and write
 * policy"): copy tokens [cold_valid, T) of an ACTIVE session into its
 * image, set cold_valid = T, return its hot blocks to the end of the free
 * list in logical order, state -> PAUSED. Tokens already in the image are
 * not rewritten. The stream first waits for the session's last append; the
 * caller orders it after any decode that still reads the session. Blocks
 * are reused only by work ordered after this pack (the pool makes later
 * allocations wait on its completion event). */
int session_pause(kv_pool *pool, int32_t sid, kv_stream_t stream);

/* Data path 2 (Section 3, "Eviction, resume and decode"): pop
 * ceil(T / bt) blocks, write the session's block-table row, copy tokens
 * [0, T) of its image into them, state -> ACTIVE, and record the session's
 * ready event on the stream. Errors: KV_ERR_BAD_STATE (not paused),
 * KV_ERR_NO_HOT_BLOCKS (nothing changes). */
int session_resume(kv_pool *pool, int32_t sid, kv_stream_t stream);

/* Event recorded after the session's last resume (NULL if none): a decode
 * stream waits on it before reading the session's blocks (Section 3,
 * "Eviction, resume and decode": a resumed session decodes once its KV is
 * back in HBM; resume overlaps other work). The event is owned by the pool
 * and stays valid until the session is destroyed. */
int session_ready_event(kv_pool *pool, int32_t sid, kv_event_t *ev);

/* State, length, capacity, cold_valid and image address of a session. */
int session_info(kv_pool *pool, int32_t sid, kv_session_info *out);

/* Host copy of a session's block-table row: up to cap entries into
 * host_row; *nblocks receives the row length. Bookkeeping; no passage (the
 * table maps a session's logical blocks to the fixed-size paged blocks of
 * Section 2, "Large Language Models"). Residency mode: an evicted block's
 * entry is -1. */
int session_block_table(kv_pool *pool, int32_t sid, int32_t *host_row, int32_t cap,
                        int32_t *nblocks);

/* Device address of a session's block-table row in the pool's table arena
 * (int32, at least ceil(max_context / block_tokens) entries; *nblocks
 * receives the number of logical blocks). Bookkeeping; no passage. For
 * callers that form their own decode batch tables on the device instead of
 * calling kv_pool_batch_tables. The pool owns the memory; the address stays
 * fixed for the pool's life. The row's entries are written by kernels on
 * the stream of the call that changed them (append, resume,
 * kv_pool_batch_reserve, a residency-mode fetch): read it on a stream
 * ordered after that call. Residency mode: the entry of a block that was
 * evicted is stale (it names a slot that may hold another session's block)
 * until the block is fetched back; use the row only while session_info
 * reports num_blocks == ceil(tokens / block_tokens). Host-logic-only pools
 * have no device arena: KV_ERR_BAD_STATE. */
int session_block_table_device(kv_pool *pool, int32_t sid, const int32_t **dev_row,
                               int32_t *nblocks);

/* Build the decode inputs of a batch of ACTIVE sessions: block_tables
 * (device int32 [B][max_blocks], entries past a row's length set to -1) and
 * seq_lens (device int32 [B]) from the pool's tables. sids is a host array
 * of B ids. */
int kv_pool_batch_tables(kv_pool *pool, const int32_t *sids, int32_t B, int32_t *block_tables,
                         int32_t max_blocks, int32_t *seq_lens, kv_stream_t stream);

/* Data path 3 for one decode step of a batch, the values written by the
 * decode kernel (decode_append_attention): each of the B distinct ACTIVE
 * sessions in sids gets position T (a block is popped when its tail block
 * is full) and T += 1; then block_tables and seq_lens are built as by
 * kv_pool_batch_tables, so seq_lens[b] counts the new token. In residency
 * mode the members' evicted blocks are fetched back first and victims come
 * only from sessions outside the batch; all members are stamped with one
 * recency time. Free-list pops go in batch order: a member's missing blocks
 * in ascending order, then its new block. The stream first waits for the
 * members' last resumes and for packs of popped blocks. Until the decode
 * has written the new tokens their slots hold stale data, so no call that
 * may pack these sessions (a pause, an eviction by a later allocation) may
 * come before it. Errors: a session twice, paused or at capacity, or
 * max_blocks too short -> KV_ERR_INVALID_ARG / KV_ERR_BAD_STATE;
 * KV_ERR_NO_HOT_BLOCKS. All or nothing. Host-logic-only pools do the
 * bookkeeping and ignore the outputs. */
int kv_pool_batch_reserve(kv_pool *pool, const int32_t *sids, int32_t B, int32_t *block_tables,
                          int32_t max_blocks, int32_t *seq_lens, kv_stream_t stream);

/* Prefetch one step ahead of decode (Section 3, "Eviction, resume and
 * decode": decode reads a known set of blocks each step, so the next step's
 * blocks are fetched ahead and flash latency stays off the step). sids: host
 * array of the B ACTIVE sessions of the NEXT decode step; busy: host array of
 * the n_busy sessions whose decode may still be running (the current step's
 * batch), or NULL with n_busy = 0. In residency mode every evicted block of
 * the next batch is fetched on `stream` (typically a migration stream, so it
 * runs beside the current step), victims coming only from sessions in
 * neither array (LRU order as for any allocation, written on eviction only
 * for tokens the image lacks); the next batch's sessions are then stamped
 * with one recency time, and each session that had blocks fetched
 * re-records its ready event on `stream`, which kv_pool_batch_reserve and
 * kv_pool_batch_tables wait on before the step reads them. The stream must
 * already be ordered after the decode steps before the current one (they
 * may have read or written the victims). Pops from the free list go member
 * by member, missing blocks in ascending order. Simple mode: nothing is ever
 * evicted, the call only validates and returns KV_OK. Errors: unknown or
 * paused session -> KV_ERR_INVALID_ARG / KV_ERR_BAD_STATE; not enough
 * evictable blocks outside both arrays -> KV_ERR_NO_HOT_BLOCKS (nothing
 * changes; the step's own batch call will then fetch what is missing, with
 * victims outside the next batch only). All or nothing. */
int kv_pool_prefetch(kv_pool *pool, const int32_t *sids, int32_t B, const int32_t *busy,
                     int32_t n_busy, kv_stream_t stream);

/* Re-run the Fisher-Yates shuffle over the current free list with a new
 * seed (scrambles where the next allocations land). */
int kv_pool_shuffle_free(kv_pool *pool, uint64_t seed);

/* Host copy of the free list (bottom to top): up to cap ids, *n = length. */
int kv_pool_free_list(kv_pool *pool, int32_t *host_out, int64_t cap, int64_t *n);

int kv_pool_get_stats(kv_pool *pool, kv_pool_stats *out);

/* Bits of the device flag word that kernels set when their own checks fire,
 * and (STALE_COUNTERS) what kv_pool_check_device finds in the workspace. */
#define KV_DEVICE_BAD_BLOCK 1      /* a block id outside the pool (access skipped)     */
#define KV_DEVICE_BAD_LENGTH 2     /* seq_len < 1 or past its table row (row skipped) */
#define KV_DEVICE_TIMEOUT 4        /* a tile wait gave up after 2 s (output undefined) */
#define KV_DEVICE_STALE_COUNTERS 8 /* split-arrival counters not at zero (reset)       */

/* Synchronise the device and read the flags that kernels set when their own
 * bounds checks fire (a block id outside the pool, a length past a table
 * row, a wait that timed out); clears them. Also checks that the decode
 * workspace's split-arrival counters are back at zero, as every decode call
 * leaves them; counters left non-zero (by decode calls that overlapped on
 * the GPU) set KV_DEVICE_STALE_COUNTERS and are reset, so later calls are
 * right again. *flags = 0 means clean; a non-zero value (KV_DEVICE_* bits)
 * makes the call return KV_ERR_DEVICE_CHECK. Bookkeeping; no passage. */
int kv_pool_check_device(kv_pool *pool, int32_t *flags);

/* Cap the migration kernels (resume-unpack, pause-pack, evictions) at
 * max_ctas CTAs of 256 threads, so that migrations running beside decode take
 * a smaller share of HBM bandwidth (Section 3, data paths: eviction and resume
 * overlap decode). 0 removes the cap (the default grid: 32 CTAs per SM).
 * Affects later calls only. */
int kv_pool_set_migration_limit(kv_pool *pool, int32_t max_ctas);

/* Test hook: make the n-th following CUDA call of this pool fail (as a
 * CUDA error) so tests can check that failing calls change nothing;
 * n <= 0 disarms. */
int kv_pool_inject_cuda_failure(kv_pool *pool, int32_t n);

/* Test hook for the decode kernel's bounded waits: with on != 0, the next
 * decode call makes warp 0 of one CTA (split 0, kv-head 0, first row) expect
 * 16 bytes more than its first tile copy delivers. Every copy still lands;
 * that one wait runs out after its 2 s limit, the kernel sets
 * KV_DEVICE_TIMEOUT, waits (bounded) for the warp's other copies and
 * finishes. That call's output for the row is undefined; the CUDA context
 * stays usable and kv_pool_check_device reports the flag. Disarms itself
 * after one call. */
int kv_pool_inject_decode_timeout(kv_pool *pool, int32_t on);

/* Test hook for the counter check: synchronises the device and sets the
 * first split-arrival counter of the workspace to 1, as a decode call that
 * overlapped another would leave it. The next kv_pool_check_device reports
 * KV_DEVICE_STALE_COUNTERS and resets it. Errors: host-logic pool ->
 * KV_ERR_BAD_STATE. */
int kv_pool_inject_stale_counter(kv_pool *pool);

/* Fixed size of the device scratch used by decode_attention_noalloc. */
#define KV_NOALLOC_SCRATCH_BYTES (48ll << 20)

/* decode_attention without any allocation. The paper has no counterpart:
 * this is a deployment variant of decode_attention.
 *
 * Who needs it: callers that cannot let a library allocate device memory,
 * such as a serving engine that reserves nearly all HBM for its own KV and
 * weight arenas up front (a library cudaMalloc could then fail, or would
 * break the engine's memory accounting), or code that cannot accept the
 * device-wide synchronisation that cudaMalloc/cudaFree may cause while
 * other streams are running. It needs no pool (creating a pool allocates).
 *
 * Same arguments and result as decode_attention, with the pool replaced by
 * `cfg`, of which only num_layers, num_q_heads, num_kv_heads, head_dim,
 * block_tokens, num_hot_blocks, hot_base and device are read. The split
 * partials live in one file-scope device array of KV_NOALLOC_SCRATCH_BYTES
 * (48 MiB) that every GPU loading the library holds until the process exits.
 * A call needs layers x B x Hq x S x 520 bytes (+256), S the split count for
 * max_blocks * block_tokens tokens (at most 16 up to 32K tokens,
 * ceil(t / 2048) beyond); larger requests fail with KV_ERR_INVALID_ARG before
 * any work.
 * It calls no cudaMalloc, cudaFree or allocating library routine.
 *
 * The first call on a device, with that device current, looks up the
 * array's device address (cudaGetSymbolAddress) and sets the decode
 * kernel's shared-memory attribute; make that first call before any stream
 * capture. All calls share the one array, and one array of split-arrival
 * counters that every call leaves at zero: calls whose work overlaps on the
 * GPU (different streams, or different host threads without ordering) race
 * and give wrong results, and counters they leave non-zero make later calls
 * wrong too; order them on one stream. Kernel bounds checks
 * keep bad block ids or lengths memory-safe but are not reported here: a
 * row whose seq_len is below 1 or beyond max_blocks * block_tokens is not
 * written at all (out keeps what it held), a block id outside the pool is
 * read as block 0 (that row's output is then wrong), and a tile wait that
 * runs out (2 s) leaves that row's output undefined. The tensor map of a
 * hot arena is encoded on its first call and kept (host memory, four
 * arenas per device). */
int decode_attention_noalloc(const kv_pool_config *cfg, int32_t layer, const void *q,
                             const int32_t *block_tables, const int32_t *seq_lens, int32_t B,
                             int32_t max_blocks, float scale, float *out, kv_stream_t stream);

/* Message of the last error on the calling thread ("" if none).
 * Bookkeeping; no passage. The string is owned by the library and valid
 * until the thread's next failing call. */
const char *kv_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* KVTIER_H */
