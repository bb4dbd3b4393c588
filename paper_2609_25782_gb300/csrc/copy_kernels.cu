// Copy kernels of the hot/cold KV tiering hot path, for sm_103a.
//
//   migrate_kernel<false>  data path 2: resume-unpack, cold image -> blocks.
//   resume_inline_kernel   the same for a resume of up to 2 048 blocks whose
//                          ids ride in the launch (it also writes the row).
//   migrate_kernel<true>   data path 4: pause-pack, blocks -> cold image,
//                          tokens [t0, T) only (write-on-evict, Section 3).
//   block_jobs_kernel<>    the same moves for explicit (slot, block, token
//                          range) lists: residency-mode evictions and fetches.
//   append_kernel          data path 3: fresh tokens into the tail blocks.
//   table_write_kernel / gather_tables_kernel: block-table bookkeeping.
//
// Hot pool: hot[NB][L][2][Hkv][bt][128] bf16. A (block, layer, K|V, head)
// run is bt rows of 256 B. The image of a session is img[L][2][Hkv][T_cap][128].
#include <cstdint>

#include "kvt_internal.h"

namespace kvt {
namespace {

// Migration copy shape, from GB300 measurements of 2..16 loads per lane and
// 4..32 CTAs per SM: 4 loads per lane over a grid of 32 CTAs per SM, one warp
// per 16-token chunk of a run, moves an 8 x 32K-token burst at the copy
// bandwidth (0.93 of it with 8 loads x 8 CTAs).
constexpr int kMigChunkTokens = 16;     // tokens per migration item (divides bt)
#ifndef KVT_MIG_UNROLL
#define KVT_MIG_UNROLL 4          // 16-byte loads in flight per lane
#endif
#ifndef KVT_MIG_CTAS_PER_SM
#define KVT_MIG_CTAS_PER_SM 32    // grid-stride CTAs of 256 threads per SM
#endif

__device__ __forceinline__ void st_out(uint4 *p, const uint4 &v) {
#ifdef KVT_MIG_STREAM_STORE
    asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y),
                 "r"(v.z), "r"(v.w)
                 : "memory");
#else
    *p = v;
#endif
}

__device__ __forceinline__ uint4 ld_stream(const uint4 *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// K3 / K4: one warp per (layer, K|V, kv-head, block) run of the token range.
// Both sides of a run are contiguous rows of 256 B; a warp moves it with
// 16-byte loads, KVT_MIG_UNROLL in flight per lane. Items are ordered run-major so
// that consecutive warps walk the image sequentially.
// The copy loop of a session's migration; block_of(j) gives logical block j's slot.
template <bool kPack, typename BlockOf>
__device__ __forceinline__ void migrate_runs(const MigArgs &a, BlockOf block_of) {
    const Shape sh = a.s;
    const int runs = sh.L * 2 * sh.Hkv;
    // Items are 16-token chunks of a run, so a 64-token block gives four
    // warps the parallelism a 16-token block gives one.
    const int q0 = a.t_begin / kMigChunkTokens;
    const int q1 = (a.t_end + kMigChunkTokens - 1) / kMigChunkTokens;
    const int nq = q1 - q0;
    const int items = runs * nq;
    const int lane = threadIdx.x & 31;
    const int nwarps = (gridDim.x * blockDim.x) >> 5;
    for (int it = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; it < items; it += nwarps) {
        const int c = it / nq;
        const int q = q0 + (it - c * nq);
        const int j = q * kMigChunkTokens / sh.bt;
        const int blk = block_of(j);
        if (blk < 0 || blk >= sh.num_blocks) {
            if (lane == 0) atomicOr(a.err, kErrBadBlock);
            continue;
        }
        const int t_lo = max(a.t_begin, q * kMigChunkTokens);
        const int t_hi = min(a.t_end, (q + 1) * kMigChunkTokens);
        uint8_t *hp = a.hot + ((static_cast<int64_t>(blk) * runs + c) * sh.bt + (t_lo - j * sh.bt)) *
                                  kRowBytes;
        uint8_t *ip = a.img + (static_cast<int64_t>(c) * a.T_cap + t_lo) * kRowBytes;
        const uint4 *src = reinterpret_cast<const uint4 *>(kPack ? hp : ip);
        uint4 *dst = reinterpret_cast<uint4 *>(kPack ? ip : hp);
        const int units = (t_hi - t_lo) * (kRowBytes / 16);
        for (int u0 = 0; u0 < units; u0 += 32 * KVT_MIG_UNROLL) {
            uint4 v[KVT_MIG_UNROLL];
#pragma unroll
            for (int k = 0; k < KVT_MIG_UNROLL; ++k) {
                const int u = u0 + k * 32 + lane;
                if (u < units) v[k] = ld_stream(src + u);
            }
#pragma unroll
            for (int k = 0; k < KVT_MIG_UNROLL; ++k) {
                const int u = u0 + k * 32 + lane;
                if (u < units) st_out(dst + u, v[k]);
            }
        }
    }
}

// K3'/K4': block-granular moves for the residency mode: one warp per
// (job, layer, K|V, kv-head) run; a job moves tokens [t0, t1) of one block.
template <bool kPack>
__global__ void __launch_bounds__(256) migrate_kernel(const MigArgs a) {
    migrate_runs<kPack>(a, [&](int j) { return a.table[j]; });
}

// Resume-unpack with the new block ids in the launch parameters: the grid
// also writes them to the session's table row (read by later work only).
__global__ void __launch_bounds__(256) resume_inline_kernel(const __grid_constant__ ResumeArgs r) {
    const int nthreads = gridDim.x * blockDim.x;
    int32_t *row = const_cast<int32_t *>(r.m.table);   // the pool's own row: writable
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < r.n; j += nthreads)
        row[j] = r.blocks[j];
    migrate_runs<false>(r.m, [&](int j) { return j < r.n ? r.blocks[j] : -1; });
}

template <bool kPack>
__global__ void __launch_bounds__(256) block_jobs_kernel(const __grid_constant__ BlockJobs a) {
    const Shape sh = a.s;
    const int runs = sh.L * 2 * sh.Hkv;
    const int cpb = sh.bt / kMigChunkTokens;      // 16-token chunks per block
    const int items = a.n * runs * cpb;
    const int lane = threadIdx.x & 31;
    const int nwarps = (gridDim.x * blockDim.x) >> 5;
    for (int it = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; it < items; it += nwarps) {
        const int jb = it / (runs * cpb);
        const int rem = it - jb * runs * cpb;
        const int c = rem / cpb;
        const int ch = rem - c * cpb;
        const BlockJob &b = a.job[jb];
        if (b.slot < 0 || b.slot >= sh.num_blocks || b.t0 < 0 || b.t1 > sh.bt) {
            if (lane == 0 && ch == 0 && c == 0) atomicOr(a.err, kErrBadBlock);
            continue;
        }
        if (!kPack && b.sid >= 0 && c == 0 && ch == 0 && lane == 0)   // a fetch: its table entry
            a.tables[static_cast<int64_t>(b.sid) * a.table_stride + b.j] = b.slot;
        const int t_lo = max(b.t0, ch * kMigChunkTokens);
        const int t_hi = min(b.t1, (ch + 1) * kMigChunkTokens);
        if (t_hi <= t_lo) continue;
        uint8_t *hp = a.hot + ((static_cast<int64_t>(b.slot) * runs + c) * sh.bt + t_lo) * kRowBytes;
        uint8_t *ip = b.img + (static_cast<int64_t>(c) * b.T_cap + static_cast<int64_t>(b.j) * sh.bt +
                               t_lo) * kRowBytes;
        const uint4 *src = reinterpret_cast<const uint4 *>(kPack ? hp : ip);
        uint4 *dst = reinterpret_cast<uint4 *>(kPack ? ip : hp);
        const int units = (t_hi - t_lo) * (kRowBytes / 16);
        for (int u0 = 0; u0 < units; u0 += 32 * KVT_MIG_UNROLL) {
            uint4 v[KVT_MIG_UNROLL];
#pragma unroll
            for (int k = 0; k < KVT_MIG_UNROLL; ++k) {
                const int u = u0 + k * 32 + lane;
                if (u < units) v[k] = ld_stream(src + u);
            }
#pragma unroll
            for (int k = 0; k < KVT_MIG_UNROLL; ++k) {
                const int u = u0 + k * 32 + lane;
                if (u < units) st_out(dst + u, v[k]);
            }
        }
    }
}

// K5: one warp per (layer, token): the token's K and V rows for all kv-heads
// are 2 x Hkv*256 contiguous bytes in the source; each 256-byte head row goes
// to its (layer, K|V, head) run of the tail block.
// One warp per (layer, token) item, items layer-major so that consecutive
// warps read k and v sequentially. A lane issues all of its 16-byte loads of
// the item (K and V rows of every kv-head) before its first store.
__global__ void __launch_bounds__(256) append_kernel(const AppendArgs a) {
    const Shape sh = a.s;
    const int items = sh.L * a.n;
    const int lane = threadIdx.x & 31;
    const int units = sh.Hkv * (kRowBytes / 16);   // 16-byte units per K (or V) token
    const int nwarps = (gridDim.x * blockDim.x) >> 5;
    for (int it = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; it < items; it += nwarps) {
        const int l = it / a.n;
        const int i = it - l * a.n;
        const int64_t t = a.pos0 + i;
        const int64_t src_off = static_cast<int64_t>(it) * sh.Hkv * kRowBytes;
        const uint4 *ks = reinterpret_cast<const uint4 *>(a.k + src_off);
        const uint4 *vs = reinterpret_cast<const uint4 *>(a.v + src_off);
        const int blk = a.table[t / sh.bt];
        const bool ok = blk >= 0 && blk < sh.num_blocks;
        if (!ok && lane == 0) atomicOr(a.err, kErrBadBlock);
        // Unit u = (kv * Hkv + g) * 16 + c lands in run (kv, g), row `slot`.
        const int slot = static_cast<int>(t % sh.bt);
        uint8_t *base = a.hot + ((static_cast<int64_t>(ok ? blk : 0) * sh.L + l) * 2 * sh.Hkv *
                                     sh.bt + slot) * kRowBytes;
        const int64_t run_bytes = static_cast<int64_t>(sh.bt) * kRowBytes;
        for (int u0 = 0; u0 < 2 * units; u0 += 32 * KVT_MIG_UNROLL) {
            uint4 v[KVT_MIG_UNROLL];
#pragma unroll
            for (int k = 0; k < KVT_MIG_UNROLL; ++k) {
                const int u = u0 + k * 32 + lane;
                if (u < 2 * units) v[k] = ld_stream(u < units ? ks + u : vs + (u - units));
            }
            if (!ok) continue;
#pragma unroll
            for (int k = 0; k < KVT_MIG_UNROLL; ++k) {
                const int u = u0 + k * 32 + lane;
                if (u < 2 * units)
                    st_out(reinterpret_cast<uint4 *>(base + (u >> 4) * run_bytes) + (u & 15), v[k]);
            }
        }
    }
}

__global__ void table_write_kernel(const __grid_constant__ TableWriteArgs a) {
    for (int i = threadIdx.x; i < a.n; i += blockDim.x) a.dst[i] = a.vals[i];
}

__global__ void gather_tables_kernel(const __grid_constant__ GatherArgs a) {
    const int r = blockIdx.x;
    if (r >= a.count) return;
    int32_t *src = a.arena + static_cast<int64_t>(a.sids[r]) * a.stride;
    int32_t *dst = a.tables + static_cast<int64_t>(a.row0 + r) * a.max_blocks;
    const int n = a.nblk[r];
    const int32_t nb = a.new_blk[r];   // a block the row just gained, not yet in the arena
    for (int e = threadIdx.x; e < a.max_blocks; e += blockDim.x)
        dst[e] = e < n ? (e == n - 1 && nb >= 0 ? nb : src[e]) : -1;
    if (threadIdx.x == 0) {
        if (nb >= 0) src[n - 1] = nb;
        a.seq_lens[a.row0 + r] = a.lens[r];
    }
}

}  // namespace

// One warp per item, 8 per CTA; at most KVT_MIG_CTAS_PER_SM per SM, or
// max_ctas when the caller caps migrations (max_ctas > 0).
static unsigned mig_grid(int64_t items, int num_sms, int max_ctas) {
    int64_t blocks = (items + 7) / 8;
    int64_t cap = static_cast<int64_t>(num_sms) * KVT_MIG_CTAS_PER_SM;
    if (max_ctas > 0 && max_ctas < cap) cap = max_ctas;
    if (blocks > cap) blocks = cap;
    return static_cast<unsigned>(blocks < 1 ? 1 : blocks);
}

cudaError_t launch_unpack(const MigArgs &a, int num_sms, int max_ctas, cudaStream_t st) {
    if (a.t_end <= a.t_begin) return cudaSuccess;
    const int64_t nq = (a.t_end + kMigChunkTokens - 1) / kMigChunkTokens - a.t_begin / kMigChunkTokens;
    migrate_kernel<false><<<mig_grid(nq * a.s.L * 2 * a.s.Hkv, num_sms, max_ctas), 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_unpack_inline(const ResumeArgs &r, int num_sms, int max_ctas, cudaStream_t st) {
    const MigArgs &a = r.m;
    if (a.t_end <= a.t_begin || r.n < 1 || r.n > kResumeInlineMax) return cudaErrorInvalidValue;
    const int64_t nq = (a.t_end + kMigChunkTokens - 1) / kMigChunkTokens - a.t_begin / kMigChunkTokens;
    resume_inline_kernel<<<mig_grid(nq * a.s.L * 2 * a.s.Hkv, num_sms, max_ctas), 256, 0, st>>>(r);
    return cudaGetLastError();
}

cudaError_t launch_pack(const MigArgs &a, int num_sms, int max_ctas, cudaStream_t st) {
    if (a.t_end <= a.t_begin) return cudaSuccess;
    const int64_t nq = (a.t_end + kMigChunkTokens - 1) / kMigChunkTokens - a.t_begin / kMigChunkTokens;
    migrate_kernel<true><<<mig_grid(nq * a.s.L * 2 * a.s.Hkv, num_sms, max_ctas), 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_append(const AppendArgs &a, int num_sms, cudaStream_t st) {
    const int64_t warps = static_cast<int64_t>(a.s.L) * a.n;
    int64_t blocks = (warps + 7) / 8;
    const int64_t cap = static_cast<int64_t>(num_sms) * KVT_MIG_CTAS_PER_SM;
    if (blocks > cap) blocks = cap;
    append_kernel<<<static_cast<unsigned>(blocks < 1 ? 1 : blocks), 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_block_jobs(const BlockJobs &a, bool pack, int num_sms, int max_ctas,
                              cudaStream_t st) {
    if (a.n <= 0) return cudaSuccess;
    const unsigned grid = mig_grid(static_cast<int64_t>(a.n) * a.s.L * 2 * a.s.Hkv *
                                       (a.s.bt / kMigChunkTokens), num_sms, max_ctas);
    if (pack)
        block_jobs_kernel<true><<<grid, 256, 0, st>>>(a);
    else
        block_jobs_kernel<false><<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_table_write(const TableWriteArgs &a, cudaStream_t st) {
    table_write_kernel<<<1, 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_gather(const GatherArgs &a, cudaStream_t st) {
    gather_tables_kernel<<<a.count, 128, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace kvt
