// Internal interface between the pool runtime (pool.cpp) and the kernels
// (decode_kernels.cu, copy_kernels.cu). Not part of the C ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace kvt {

constexpr int kHeadDim = 128;     // D; one token row of one head is 256 B
constexpr int kRowBytes = kHeadDim * 2;
constexpr int kTileTokens = 16;   // tokens per decode tile (one mma M)
constexpr int kMaxGroup = 8;      // Hq / Hkv handled by one CTA

// Device-side check flags (OR-ed into the pool's error word).
constexpr int32_t kErrBadBlock = 1;    // block id outside the pool
constexpr int32_t kErrBadLength = 2;   // seq_len < 1 or past its table row
constexpr int32_t kErrTimeout = 4;     // an mbarrier wait gave up

// Split-KV plan. A pure function of the session length, so a session's
// result never depends on batch composition or placement: split s covers
// tiles [s*split_tiles, (s+1)*split_tiles) of the ceil(T/16) 16-token tiles.
// split_tiles = clamp(ceil(tiles / 16), KVT_SPLIT_MIN_TILES, KVT_SPLIT_MAX_TILES).
// The defaults, 64..128 tiles (1 024 tokens up to 16K-token sessions, growing
// to 2 048 at 32K), come from GB300 measurements of 8..128-tile variants:
// long splits leave few partials to merge, while 1 024-token splits keep
// enough CTAs for the smaller batches of an agentic trace.
#ifndef KVT_SPLIT_MIN_TILES
#define KVT_SPLIT_MIN_TILES 64
#endif
#ifndef KVT_SPLIT_MAX_TILES
#define KVT_SPLIT_MAX_TILES 128
#endif
#ifndef KVT_SPLIT_TARGET
#define KVT_SPLIT_TARGET 16       // splits per (session, kv-head) while the clamp is inactive
#endif
__host__ __device__ inline int tiles_of(int T) { return (T + kTileTokens - 1) / kTileTokens; }
__host__ __device__ inline int split_tiles(int T) {
    int s = (tiles_of(T) + KVT_SPLIT_TARGET - 1) / KVT_SPLIT_TARGET;
    return s < KVT_SPLIT_MIN_TILES ? KVT_SPLIT_MIN_TILES
                                   : (s > KVT_SPLIT_MAX_TILES ? KVT_SPLIT_MAX_TILES : s);
}
__host__ __device__ inline int num_splits(int T) {
    int st = split_tiles(T);
    return (tiles_of(T) + st - 1) / st;
}
// Upper bound of num_splits(T) for T <= max_tokens. Below target*min tiles
// the split is min tiles (ceil(tiles/min) splits, fewer than the target);
// while the clamp is inactive there are at most `target`; above target*max
// tiles, ceil(tiles/max).
inline int max_splits_for(int64_t max_tokens) {
    const int64_t tiles = (max_tokens + kTileTokens - 1) / kTileTokens;
    const int64_t at_max = (tiles + KVT_SPLIT_MAX_TILES - 1) / KVT_SPLIT_MAX_TILES;
    int64_t at_min = (tiles + KVT_SPLIT_MIN_TILES - 1) / KVT_SPLIT_MIN_TILES;
    if (at_min > KVT_SPLIT_TARGET) at_min = KVT_SPLIT_TARGET;
    return (int)(at_max > at_min ? at_max : at_min);
}

struct Shape {
    int32_t L, Hq, Hkv, bt;
    int64_t num_blocks;
};

struct DecodeArgs {
    const uint16_t *q;        // [nl][B][Hq][D] bf16
    const int32_t *tables;    // [B][max_blocks]
    const int32_t *seq_lens;  // [B]
    float *out;               // [nl][B][Hq][D], fp32 or (out_bf16) bf16
    float *part_o;            // [nl*B][Hq][max_splits][D]
    float *part_ml;           // [nl*B][Hq][max_splits][2]
    int32_t *counters;        // [nl*B][Hkv] split arrivals; zero between calls
    int32_t merge_max_splits; // sessions of 2..this many splits merge in the split kernel
    int32_t *err;
    int32_t B, max_blocks, layer0, nlayers, max_splits;
    float scale_log2;         // scale * log2(e)
    int32_t out_bf16;         // 1: out holds bf16 (round to nearest even)
    // Fused append (data path 3): when k_new is set, token seq_lens[b]-1 of
    // each row arrives with the call, bf16 [nl][B][Hkv][D] each, and is
    // written into its reserved pool slot as well as attended to.
    const uint16_t *k_new, *v_new;
    uint16_t *hot;            // pool base, written only when k_new is set
    int32_t inject_extra_tx;  // test hook: extra bytes expected on one tile (0 normally)
    Shape s;
};

struct MigArgs {
    const int32_t *table;     // session's block-table row (device)
    uint8_t *hot;
    uint8_t *img;
    int64_t T_cap;            // image rows per (layer, K|V, kv-head) run
    int32_t t_begin, t_end;   // tokens to move
    int32_t *err;
    Shape s;
};

// A resume whose new block ids ride in the launch: the kernel writes the
// session's table row itself and needs no prior table-write launch.
constexpr int kResumeInlineMax = 2048;   // blocks (32K tokens at bt = 16)
struct ResumeArgs {
    MigArgs m;                // m.table: the session's device row, written here
    int32_t n;                // blocks in the row
    int32_t pad;
    int32_t blocks[kResumeInlineMax];
};

struct AppendArgs {
    const uint8_t *k, *v;     // [L][n][Hkv][D] bf16
    const int32_t *table;
    uint8_t *hot;
    int64_t pos0;
    int32_t n;
    int32_t *err;
    Shape s;
};

// One block move between a hot slot and a session image: tokens [t0, t1) of
// logical block j (all layers, K and V, all kv-heads).
struct BlockJob {
    uint8_t *img;             // the session's image base
    int32_t T_cap;            // image rows per (layer, K|V, kv-head) run (contexts <= 2^30)
    int32_t sid;              // a fetch: the session whose table entry j becomes `slot`; -1: none
    int32_t slot, j, t0, t1;
};
constexpr int kBlockJobsMax = 960;   // keeps the parameter block under 32 KB
struct BlockJobs {
    uint8_t *hot;
    int32_t *err;
    int32_t *tables;          // the pool's table arena (fetch jobs write their entry)
    int64_t table_stride;
    Shape s;
    int32_t n;
    int32_t pad;
    BlockJob job[kBlockJobsMax];
};

constexpr int kTableWriteMax = 2048;
struct TableWriteArgs {
    int32_t *dst;
    int32_t n;
    int32_t vals[kTableWriteMax];
};

constexpr int kGatherMax = 512;
struct GatherArgs {
    int32_t *arena;           // [max_sessions][stride]
    int64_t stride;
    int32_t *tables;          // [B][max_blocks]
    int32_t *seq_lens;
    int32_t max_blocks;
    int32_t count;            // rows written by this launch
    int32_t row0;             // first batch row of this launch
    int32_t sids[kGatherMax];
    int32_t lens[kGatherMax];
    int32_t nblk[kGatherMax];
    int32_t new_blk[kGatherMax];   // >= 0: also store it as the row's last entry (nblk-1)
};

// Host launchers (decode_kernels.cu, copy_kernels.cu). Each returns the launch's CUDA status.
// The decode kernel's tensor map of the hot pool: rows of 128 bf16, and
// run_rows (Hkv * bt) rows between a (block, layer) K run and its V run.
bool encode_hot_tensor_map(CUtensorMap *map, void *hot_base, int64_t rows, int64_t run_rows,
                           const char **why);
cudaError_t prepare_kernels();  // per-device function attributes
// overlap_previous: launch the split kernel as a programmatic dependent of the
// previous kernel on the stream (see decode_attention_ex). num_sms sizes the
// split kernel's tile rings to the grid.
cudaError_t launch_decode(const CUtensorMap &map, const DecodeArgs &a, int num_sms,
                          cudaStream_t st, bool overlap_previous);
// max_ctas > 0 caps the migration grids (kv_pool_set_migration_limit).
cudaError_t launch_unpack(const MigArgs &a, int num_sms, int max_ctas, cudaStream_t st);
cudaError_t launch_unpack_inline(const ResumeArgs &r, int num_sms, int max_ctas, cudaStream_t st);
cudaError_t launch_pack(const MigArgs &a, int num_sms, int max_ctas, cudaStream_t st);
cudaError_t launch_append(const AppendArgs &a, int num_sms, cudaStream_t st);
cudaError_t launch_block_jobs(const BlockJobs &a, bool pack, int num_sms, int max_ctas,
                              cudaStream_t st);
cudaError_t launch_table_write(const TableWriteArgs &a, cudaStream_t st);
cudaError_t launch_gather(const GatherArgs &a, cudaStream_t st);

// Sets the message returned by kv_last_error() on this thread (pool.cpp).
void set_last_error(const char *msg);

}  // namespace kvt
