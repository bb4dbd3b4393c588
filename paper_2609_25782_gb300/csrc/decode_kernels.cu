// Decode-attention kernels of the hot/cold KV tiering hot path, for sm_103a.
//
//   decode_split_kernel    data path 1 (Section 3): split-KV paged GQA decode
//                          attention with an fp32 online softmax; KV tiles are
//                          staged by TMA (cp.async.bulk.tensor, 128-byte
//                          swizzle) into a per-warp mbarrier ring, and the
//                          group-by-tile products run on mma.sync bf16.
//                          In a long grid, the last CTA of a kv-head of a
//                          session of at most 4 splits to finish merges them
//                          (log-sum-exp in a fixed order).
//   decode_combine_small_kernel, decode_combine_kernel
//                          the same merge for the other multi-split sessions
//                          (one warp per query head from registers, up to 16
//                          splits; else four warps per head), launched as a
//                          programmatic dependent of the split kernel.
//
// Hot pool: hot[NB][L][2][Hkv][bt][128] bf16. A (block, layer, K|V, head)
// run is bt rows of 256 B, row = ((blk*L + l)*2 + kv)*Hkv + g)*bt + slot. The
// decode kernel views the pool as a 4-D tensor (64 columns, row, column half,
// K|V) and loads one box per 16-token tile: its 16 K rows and 16 V rows.
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include "kvt_internal.h"

namespace kvt {
namespace {

#ifndef KVT_STAGES
#define KVT_STAGES 2   // 4 warps x 2 x 8 KiB: 3 CTAs (24 tiles in flight) per SM
#endif
constexpr int kCombineWarps = 4;
// The merge of a session's splits folds four chains (contiguous quarters of
// the splits, in split order) and then merges the chains in order; that order
// depends on the split count only, whichever kernel runs it. One warp merges
// up to kRegMergeMax splits from registers (four per chain); the split kernel
// merges sessions of up to kSplitKernelMerge splits itself in long grids.
constexpr int kMergeChains = 4;
constexpr int kRegMergeMax = 16;
constexpr int kSplitKernelMerge = 4;
static_assert(kCombineWarps == kMergeChains && kRegMergeMax == kMergeChains * 4 &&
                  kSplitKernelMerge <= kRegMergeMax,
              "four splits per chain in a register merge, one chain per combine warp");
constexpr int kTileBytes = 8192;           // K 4 KiB + V 4 KiB
constexpr int kHalfBytes = 2048;           // 16 rows x 128 B (64 dims)
// The plan of one split: its tiles are dealt round robin to kAccs running
// softmax states (accumulator v takes tiles v, v + kAccs, ...), which merge
// in the order v = 0 .. kAccs-1 at the end. That plan fixes the result; how
// the accumulators map to warps is a launch choice:
//   <4 warps, KVT_STAGES slots>  3 CTAs per SM; a warp owns accumulators w
//                                and w + 4 and alternates between them, so
//                                consecutive tiles of a warp are independent
//   <4 warps, 3 slots>           2 CTAs per SM
//   <8 warps, 3 slots>           1 CTA per SM (small grids): one accumulator
//                                per warp, twice the warps per SM
// Each SM keeps about 24 tiles in flight whatever the variant, and every
// variant gives bit-identical results.
constexpr int kAccs = 8;
// Lazy softmax maximum: the reference moves when a logit exceeds it by more
// than this many powers of two (P then stays at most 2^8 = 256).
constexpr float kLazyLog2 = 8.f;
#ifndef KVT_WAVE_MARGIN
#define KVT_WAVE_MARGIN 0.1   // last-wave fill gain that moves a grid to 2 CTAs per SM
#endif
constexpr int kWarpsNarrow = 4, kWarpsWide = 8;
constexpr int kStagesFull = KVT_STAGES;    // 3 CTAs per SM
constexpr int kStagesHalf = 3;             // 2 CTAs per SM
constexpr int kStagesOne = 3;              // 1 CTA per SM (8 warps)
__host__ __device__ constexpr int decode_smem(int warps, int stages) {
    return warps * stages * kTileBytes + 1024 + 256;   // rings, alignment, barriers
}
static_assert(kWarpsWide * kStagesOne * 8 <= 256, "mbarriers must fit their 256-byte area");
static_assert(kWarpsNarrow * kStagesHalf * 8 <= 256, "mbarriers must fit their 256-byte area");
constexpr unsigned long long kWaitLimitNs = 2000000000ull;   // 2 s

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait for a phase with a wall-clock limit; false means the limit expired.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (global_ns() - t0 > kWaitLimitNs) return false;
    }
    return true;
}

// One tile: the box (64 columns, 16 rows, 2 column halves, K and V) of the
// hot pool's 4-D view, starting at K row `row`.
__device__ __forceinline__ void tma_load_tile(uint32_t dst, const CUtensorMap *map, int row,
                                              uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(row), "r"(0), "r"(0), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1,
                                          uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// D = A(16x16 bf16, row) * B(16x8 bf16, col) + D, fp32 accumulate.
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t movmatrix_t(uint32_t x) {
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi, float &rlo, float &rhi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    rlo = __low2float(v);
    rhi = __high2float(v);
    return *reinterpret_cast<uint32_t *>(&v);
}

// Byte offset, inside a 16-row x 128-byte box written with the 128-byte
// swizzle, of 16-byte unit `c` (0..7) of row `r`.
__device__ __forceinline__ uint32_t swz(int r, int c) {
    return static_cast<uint32_t>(r * 128 + ((c ^ (r & 7)) << 4));
}

// Acquire-release add at GPU scope: orders this CTA's partial writes (made
// visible to thread 0 by the preceding barrier) before its arrival, and the
// last arrival's reads of the other partials after it.
__device__ __forceinline__ int arrive(int32_t *counter) {
    int prev;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;"
                 : "=r"(prev)
                 : "l"(counter)
                 : "memory");
    return prev;
}

// One step of a running log-sum-exp merge: fold the partial (m, l) = v with
// accumulator o into (m, lsum, acc). The roundings are spelled out (one
// product, then one fused multiply-add), so that the split kernel and the
// combine kernel, which both run this, give the same bits.
__device__ __forceinline__ float fold(float x, float c, float w, float y) {
    return __fmaf_rn(x, c, __fmul_rn(w, y));
}
__device__ __forceinline__ void lse_step(float &m, float &lsum, float4 &acc, const float2 v,
                                         const float4 o) {
    const float mn = fmaxf(m, v.x);
    const float c = ex2(m - mn);                   // rescale what is summed so far
    const float w = ex2(v.x - mn);
    m = mn;
    lsum = fold(lsum, c, w, v.y);
    acc.x = fold(acc.x, c, w, o.x);
    acc.y = fold(acc.y, c, w, o.y);
    acc.z = fold(acc.z, c, w, o.z);
    acc.w = fold(acc.w, c, w, o.w);
}

// The chains' states merged in chain order and normalised; lane t writes
// dims 4t..4t+3 of output row `row`.
__device__ __forceinline__ void merge_chains_store(const DecodeArgs &a, int64_t row, int lane,
                                                   const float (&m)[kMergeChains],
                                                   const float (&l)[kMergeChains],
                                                   const float4 (&acc)[kMergeChains]) {
    float M = m[0];
#pragma unroll
    for (int q = 1; q < kMergeChains; ++q) M = fmaxf(M, m[q]);
    float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
    float lt = 0.f;
#pragma unroll
    for (int q = 0; q < kMergeChains; ++q) {
        const float c = ex2(m[q] - M);             // an empty chain has m = -inf: c = 0
        r.x = __fmaf_rn(c, acc[q].x, r.x);
        r.y = __fmaf_rn(c, acc[q].y, r.y);
        r.z = __fmaf_rn(c, acc[q].z, r.z);
        r.w = __fmaf_rn(c, acc[q].w, r.w);
        lt = __fmaf_rn(c, l[q], lt);
    }
    const float inv = __frcp_rn(lt);
    const float4 y = make_float4(__fmul_rn(r.x, inv), __fmul_rn(r.y, inv), __fmul_rn(r.z, inv),
                                 __fmul_rn(r.w, inv));
    if (a.out_bf16) {
        float r0, r1;
        uint2 pk;
        pk.x = pack_bf16(y.x, y.y, r0, r1);
        pk.y = pack_bf16(y.z, y.w, r0, r1);
        reinterpret_cast<uint2 *>(reinterpret_cast<uint16_t *>(a.out) + row * kHeadDim)[lane] = pk;
    } else {
        reinterpret_cast<float4 *>(a.out + row * kHeadDim)[lane] = y;
    }
}

// The merge of one query head's ns (2..16) split partials by one warp. Every
// load is issued before the first is used (indices clamped into the row, so
// the loads need no guard): lane t loads split t's (m, l), shared by shuffle,
// and each lane its 4 dims of every split's accumulator. The partials come
// from L2 (.cg), written there by other SMs.
__device__ __forceinline__ void merge_head_regs(const DecodeArgs &a, int64_t row, int ns,
                                                     int lane) {
    const int64_t base = row * a.max_splits;
    const float2 mine = __ldcg(reinterpret_cast<const float2 *>(a.part_ml) + base +
                               min(lane, ns - 1));
    const float4 *po = reinterpret_cast<const float4 *>(a.part_o + base * kHeadDim) + lane;
    float4 o[kMergeChains][4];
    int s0[kMergeChains], n[kMergeChains];
#pragma unroll
    for (int q = 0; q < kMergeChains; ++q) {
        s0[q] = (q * ns) / kMergeChains;
        n[q] = ((q + 1) * ns) / kMergeChains - s0[q];
#pragma unroll
        for (int i = 0; i < 4; ++i) o[q][i] = __ldcg(po + min(s0[q] + i, ns - 1) * (kHeadDim / 4));
    }
    float m[kMergeChains], l[kMergeChains];
    float4 acc[kMergeChains];
#pragma unroll
    for (int q = 0; q < kMergeChains; ++q) {
        m[q] = -INFINITY;
        l[q] = 0.f;
        acc[q] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int sp = min(s0[q] + i, ns - 1);
            const float2 v = make_float2(__shfl_sync(0xffffffffu, mine.x, sp),
                                         __shfl_sync(0xffffffffu, mine.y, sp));
            if (i < n[q]) lse_step(m[q], l[q], acc[q], v, o[q][i]);
        }
    }
    merge_chains_store(a, row, lane, m, l, acc);
}

// ---------------------------------------------------------------------------
// K1: one CTA = (split s, kv-head g, layer-batch row lb = li*B + b).
// The split's tiles go round robin to kAccs = 8 accumulators; warp w of the
// kWarps consumes tiles w, w + kWarps, ... through its own ring of kStages
// 8 KiB slots, tile k of the warp feeding its accumulator k % (8 / kWarps).
// Per tile (16 tokens):
//   S^T[16 tok x 8 heads] = K[16 x 128] . Q^T       8 x mma m16n8k16
//   online softmax over tokens (columns = heads)
//   O^T[128 x 8] += V^T[128 x 16] . P^T[16 x 8]     8 x mma, P^T via movmatrix
// The accumulators merge in shared memory in accumulator order; a one-split
// session writes its normalised output, others write (m, l, acc) partials,
// which the group's last CTA to finish merges when the launch allows it
// (a.merge_max_splits), else the combine kernel.
// ---------------------------------------------------------------------------
struct AccState {
    float m0, m1;   // running max, heads 2(lane%4) and +1 (log2 units)
    float l0, l1;   // this lane's share of the normaliser
    float o[8][4];  // O^T fragments
};

template <int kWarps, int kStages>
__global__ void __launch_bounds__(kWarps * 32, kWarps == kWarpsNarrow && kStages == kStagesFull ? 3 : 1)
    decode_split_kernel(const __grid_constant__ CUtensorMap map, const DecodeArgs a) {
    constexpr int kA = kAccs / kWarps;   // accumulators per warp
    static_assert(kA * kWarps == kAccs, "accumulators divide among the warps");
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kWarps * kStages * kTileBytes);

    // The grid is (splits, kv-heads, rows); its blocks go out in linear order,
    // read here head-fastest so the CTAs of one split's kv-heads, whose runs
    // sit side by side in each block, start together (measured slightly
    // faster than split-fastest; the work of each CTA is the same).
    const int64_t lin = blockIdx.x + static_cast<int64_t>(gridDim.x) *
                                         (blockIdx.y + static_cast<int64_t>(gridDim.y) * blockIdx.z);
    const int g = static_cast<int>(lin % gridDim.y);
    const int split = static_cast<int>((lin / gridDim.y) % gridDim.x);
    const int lb = static_cast<int>(lin / (static_cast<int64_t>(gridDim.y) * gridDim.x));
    const int b = lb % a.B;
    const int li = lb / a.B;
    const int l = a.layer0 + li;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const Shape sh = a.s;
    const int G = sh.Hq / sh.Hkv;

    // The combine kernel, or the next call launched with the overlap option,
    // may be scheduled once every CTA of this grid has started; it still
    // waits for this grid to finish before reading.
    asm volatile("griddepcontrol.launch_dependents;");
    const int32_t *trow = a.tables + static_cast<int64_t>(b) * a.max_blocks;
    // Tables at most KVT_SPLIT_TARGET x KVT_SPLIT_MIN_TILES tiles wide split
    // every session every KVT_SPLIT_MIN_TILES tiles, so this warp's tiles are
    // known before T: their block ids load alongside T instead of after it.
    // Lanes past the session's tiles may read table entries past its blocks
    // (never used).
    constexpr int kMinWarpTiles = KVT_SPLIT_MIN_TILES / kWarps;
    const bool fixed_split = split_tiles(a.max_blocks * sh.bt) == KVT_SPLIT_MIN_TILES;
    int early_blk = 0;
    if (fixed_split && lane < kMinWarpTiles) {
        const int j = (split * KVT_SPLIT_MIN_TILES + warp + lane * kWarps) * kTileTokens / sh.bt;
        if (j < a.max_blocks) early_blk = trow[j];
    }
    const int T = a.seq_lens[b];
    if (T < 1 || T > a.max_blocks * sh.bt) {
        if (split == 0 && g == 0 && threadIdx.x == 0) atomicOr(a.err, kErrBadLength);
        return;
    }
    const int nsplit = num_splits(T);
    if (split >= nsplit) return;
    const int st = split_tiles(T);
    const int tile0 = split * st;
    const int tile1 = min(tiles_of(T), tile0 + st);
    const int my_tiles = (tile1 - tile0 - warp + kWarps - 1) / kWarps;  // may be <= 0

    uint8_t *ring = smem + warp * kStages * kTileBytes;
    const uint32_t ring_s = smem_u32(ring);
    const uint32_t bar0 = smem_u32(bars + warp * kStages);
    const int chunk_rows = sh.Hkv * sh.bt;   // rows between K and V runs

    // Block ids of this warp's tiles, fetched together up front: lane t
    // holds the block of the warp's tile t, so no table load waits in front
    // of a tile copy (one CTA per SM has no other warps to hide it behind).
    static_assert((KVT_SPLIT_MAX_TILES + kWarps - 1) / kWarps <= 32,
                  "a warp's tiles of one split must fit one block id per lane");
    static_assert(KVT_SPLIT_MIN_TILES % kWarps == 0, "whole tiles per warp");
    int lane_blk = early_blk;
    if (!fixed_split && lane < my_tiles)
        lane_blk = trow[(tile0 + warp + lane * kWarps) * kTileTokens / sh.bt];

    if (lane == 0) {
        for (int i = 0; i < kStages; ++i) mbar_init(bar0 + 8 * i, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncwarp();

    // Producer step (lane 0): tile k of this warp, in block blk, into slot
    // k % kStages.
    auto issue = [&](int k, int blk) {
        const int ti = tile0 + warp + k * kWarps;
        const int tok = ti * kTileTokens;
        const int j = tok / sh.bt;
        if (blk < 0 || blk >= sh.num_blocks) {
            atomicOr(a.err, kErrBadBlock);
            blk = 0;
        }
        const int rowk = ((blk * sh.L + l) * 2 * sh.Hkv + g) * sh.bt + (tok - j * sh.bt);
        const uint32_t slot = ring_s + (k % kStages) * kTileBytes;
        const uint32_t bar = bar0 + 8 * (k % kStages);
        // inject_extra_tx (a test of the bounded wait, 0 in normal calls): this
        // one barrier then never completes its phase, although every copy lands.
        const bool injected = k == 0 && warp == 0 && split == 0 && g == 0 && lb == 0;
        mbar_expect_tx(bar, kTileBytes + (injected ? a.inject_extra_tx : 0));
        tma_load_tile(slot, &map, rowk, bar);
    };
    // The block of tile k, for every lane (k < 32 wherever it is used).
    auto blk_of = [&](int k) { return __shfl_sync(0xffffffffu, lane_blk, k & 31); };
#pragma unroll
    for (int k = 0; k < kStages; ++k) {
        const int blk = blk_of(k);
        if (lane == 0 && k < my_tiles) issue(k, blk);
    }

    // Everything above reads only the hot pool, the block table and seq_lens.
    // When this grid is launched as a programmatic dependent (the caller's
    // overlap option) it may run while the previous decode call drains; Q is
    // read, and partials/outputs written, only after that call completes.
    asm volatile("griddepcontrol.wait;" ::: "memory");

    // Q^T fragments (mma B operand): head n = lane/4 of the group, dims
    // 16*ks + 2*(lane%4) + {0,1} and +8.
    uint32_t qb[8][2];
    {
        const int n = lane >> 2;
        const bool live = n < G;
        const uint32_t *qrow = reinterpret_cast<const uint32_t *>(
            a.q + ((static_cast<int64_t>(li) * a.B + b) * sh.Hq + g * G + (live ? n : 0)) *
                      kHeadDim);
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
            qb[ks][0] = live ? qrow[ks * 8 + (lane & 3)] : 0u;
            qb[ks][1] = live ? qrow[ks * 8 + 4 + (lane & 3)] : 0u;
        }
    }

    AccState acc_state[kA];
#pragma unroll
    for (int i = 0; i < kA; ++i) {
        acc_state[i].m0 = acc_state[i].m1 = -INFINITY;
        acc_state[i].l0 = acc_state[i].l1 = 0.f;
#pragma unroll
        for (int r = 0; r < 8; ++r)
            acc_state[i].o[r][0] = acc_state[i].o[r][1] = acc_state[i].o[r][2] = acc_state[i].o[r][3] = 0.f;
    }
    const float sl = a.scale_log2;
    int fail_k = -1;

    // ldmatrix lane roles. K (A operand, row-major): row = token.
    const int krow = (lane & 7) + ((lane >> 3) & 1) * 8;
    const int khi = lane >> 4;
    // V (A operand of O^T, loaded transposed): row = token.
    const int vrow = (lane & 7) + (lane >> 4) * 8;
    const int vhi = (lane >> 3) & 1;

    // Fused append: token T-1 arrives with this call. Its K and V rows
    // replace whatever the copy brought for that slot of tile k and are
    // stored to the reserved pool slot. Lanes 0-15 move K, 16-31 V, 16 B each.
    auto splice_new = [&](int k, int tok_base) {
        const int r = T - 1 - tok_base;
        const int u = lane & 15;
        const int isv = lane >> 4;
        const uint4 val = *reinterpret_cast<const uint4 *>(
            (isv ? a.v_new : a.k_new) +
            ((static_cast<int64_t>(li) * a.B + b) * sh.Hkv + g) * kHeadDim + u * 8);
        *reinterpret_cast<uint4 *>(ring + (k % kStages) * kTileBytes + isv * 2 * kHalfBytes +
                                   (u >> 3) * kHalfBytes + swz(r, u & 7)) = val;
        const int j = (T - 1) / sh.bt;
        const int blk = trow[j];
        if (blk >= 0 && blk < sh.num_blocks) {   // a bad id was flagged by the copy
            const int64_t row =
                ((static_cast<int64_t>(blk) * sh.L + l) * 2 * sh.Hkv + g) * sh.bt +
                (T - 1 - j * sh.bt) + isv * chunk_rows;
            *reinterpret_cast<uint4 *>(a.hot + row * kHeadDim + u * 8) = val;
        }
        // The slot is refilled by the async proxy later.
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
    };
    // One k-step (16 dims) of S^T = K . Q^T into acc.
    auto qk_step = [&](uint32_t slot, int ks, float (&acc)[4]) {
        uint32_t r0, r1, r2, r3;
        const int u = 2 * ks + khi;
        ldsm_x4(slot + (u >> 3) * kHalfBytes + swz(krow, u & 7), r0, r1, r2, r3);
        mma_bf16(acc, r0, r1, r2, r3, qb[ks][0], qb[ks][1]);
    };
    // Logits in log2 units; tokens at or past T are -inf.
    auto logits = [&](const float (&sa)[4], const float (&sb)[4], int tok_base, float (&x)[4]) {
        const bool v0 = tok_base + (lane >> 2) < T;
        const bool v1 = tok_base + (lane >> 2) + 8 < T;
        x[0] = v0 ? (sa[0] + sb[0]) * sl : -INFINITY;
        x[1] = v0 ? (sa[1] + sb[1]) * sl : -INFINITY;
        x[2] = v1 ? (sa[2] + sb[2]) * sl : -INFINITY;
        x[3] = v1 ? (sa[3] + sb[3]) * sl : -INFINITY;
    };
    // Last, partial tile: slots past T may hold anything (NaN); P is 0 there
    // but 0 * NaN is not, so clear those V rows of tile k.
    auto clear_tail_v = [&](int k, int tok_base) {
        if (tok_base + kTileTokens > T) {
            const int first_bad = T - tok_base;
            const int units = (kTileTokens - first_bad) * 16;
            uint8_t *vp = ring + (k % kStages) * kTileBytes + 2 * kHalfBytes;
            for (int u = lane; u < units; u += 32) {
                const int r = first_bad + (u >> 4);
                const int h = (u >> 3) & 1;
                *reinterpret_cast<uint4 *>(vp + h * kHalfBytes + r * 128 + (u & 7) * 16) =
                    make_uint4(0u, 0u, 0u, 0u);
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
        }
    };
    auto tile_base = [&](int k) { return (tile0 + warp + k * kWarps) * kTileTokens; };

    // One tile into accumulator s: scores, softmax, O^T += V^T . P^T.
    // False: its wait timed out.
    auto one_tile = [&](int k, AccState &s) -> bool {
        const uint32_t slot = ring_s + (k % kStages) * kTileBytes;
        if (!mbar_wait(bar0 + 8 * (k % kStages), (k / kStages) & 1)) return false;
        const int tok_base = tile_base(k);
        if (a.k_new != nullptr && tok_base + kTileTokens >= T) splice_new(k, tok_base);

        // S^T = K . Q^T, two accumulators to shorten the mma chain.
        float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int ks = 0; ks < 8; ks += 2) {
            qk_step(slot, ks, sa);
            qk_step(slot, ks + 1, sb);
        }
        float x[4];
        logits(sa, sb, tok_base, x);
        // Online-softmax step with a lazy maximum: the reference point m moves
        // only when a logit of the tile exceeds it by more than kLazyLog2 (the
        // first tile always does, m starting at -inf); otherwise P = 2^(x - m)
        // stays at most 2^kLazyLog2 and neither m, l nor the accumulator are
        // rescaled. When it moves, m becomes the exact running maximum (a
        // quad-shuffle reduction over the tile's columns) and l and O are
        // rescaled by 2^(m_old - m_new). P is rounded to bf16, as the PV
        // product sees it. The decision is the warp's and depends only on the
        // tile's logits and the state, so every launch variant takes it alike.
        const bool grow = (x[0] > s.m0 + kLazyLog2) | (x[2] > s.m0 + kLazyLog2) |
                          (x[1] > s.m1 + kLazyLog2) | (x[3] > s.m1 + kLazyLog2);
        if (__any_sync(0xffffffffu, grow)) {
            float mx0 = fmaxf(x[0], x[2]), mx1 = fmaxf(x[1], x[3]);
#pragma unroll
            for (int off = 4; off < 32; off <<= 1) {
                mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
                mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
            }
            const float mn0 = fmaxf(s.m0, mx0), mn1 = fmaxf(s.m1, mx1);
            const float al0 = ex2(s.m0 - mn0), al1 = ex2(s.m1 - mn1);
            s.m0 = mn0;
            s.m1 = mn1;
            s.l0 *= al0;
            s.l1 *= al1;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                s.o[i][0] *= al0;
                s.o[i][1] *= al1;
                s.o[i][2] *= al0;
                s.o[i][3] *= al1;
            }
        }
        float q0, q1, q2, q3;
        const uint32_t p01 = pack_bf16(ex2(x[0] - s.m0), ex2(x[1] - s.m1), q0, q1);
        const uint32_t p23 = pack_bf16(ex2(x[2] - s.m0), ex2(x[3] - s.m1), q2, q3);
        s.l0 += q0 + q2;
        s.l1 += q1 + q3;
        const uint32_t pb0 = movmatrix_t(p01);   // P^T tokens 0-7  -> B fragment
        const uint32_t pb1 = movmatrix_t(p23);   // P^T tokens 8-15
        clear_tail_v(k, tok_base);
        const uint32_t vslot = slot + 2 * kHalfBytes;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            uint32_t r0, r1, r2, r3;
            const int u = 2 * i + vhi;
            ldsm_x4_t(vslot + (u >> 3) * kHalfBytes + swz(vrow, u & 7), r0, r1, r2, r3);
            mma_bf16(s.o[i], r0, r1, r2, r3, pb0, pb1);
        }
        __syncwarp();
        const int nblk = blk_of(k + kStages);
        if (lane == 0 && k + kStages < my_tiles) issue(k + kStages, nblk);
        return true;
    };

    // Consecutive tiles of a warp feed different accumulators (kA = 2), so
    // the second tile's work does not wait for the first tile's products.
    for (int k = 0; k < my_tiles; k += kA) {
        if (!one_tile(k, acc_state[0])) {
            fail_k = k;
            break;
        }
        if constexpr (kA == 2) {
            if (k + 1 < my_tiles && !one_tile(k + 1, acc_state[1])) {
                fail_k = k + 1;
                break;
            }
        }
    }

    if (fail_k >= 0) {
        if (lane == 0) atomicOr(a.err, kErrTimeout);
        // Tiles fail_k .. fail_k+kStages-1 were issued and not consumed: wait
        // (again bounded) for them so no copy lands after the CTA exits.
        for (int k = fail_k; k < fail_k + kStages && k < my_tiles; ++k)
            mbar_wait(bar0 + 8 * (k % kStages), (k / kStages) & 1);
    }

    // Accumulator states -> this warp's own ring (all of its loads have
    // completed): accumulator v = warp + kWarps * i at float offset
    // i * kAccFloats of warp (v % kWarps)'s ring.
    constexpr int kOStride = kHeadDim + 4;   // floats per head row (bank skew)
    constexpr int kAccFloats = kMaxGroup * kOStride + 2 * kMaxGroup;   // O rows, m[8], l[8]
    static_assert(kA * kAccFloats * 4 <= kStages * kTileBytes, "states fit the ring");
#pragma unroll
    for (int i = 0; i < kA; ++i) {
        AccState &s = acc_state[i];
        // Normaliser: reduce the per-lane shares over the 8 lanes of a column.
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            s.l0 += __shfl_xor_sync(0xffffffffu, s.l0, off);
            s.l1 += __shfl_xor_sync(0xffffffffu, s.l1, off);
        }
        float *ws = reinterpret_cast<float *>(ring) + i * kAccFloats;
        float *wm = ws + kMaxGroup * kOStride;   // m[8], l[8]
        const int h0 = 2 * (lane & 3);
#pragma unroll
        for (int r = 0; r < 8; ++r) {
            const int d = 16 * r + (lane >> 2);
            ws[h0 * kOStride + d] = s.o[r][0];
            ws[(h0 + 1) * kOStride + d] = s.o[r][1];
            ws[h0 * kOStride + d + 8] = s.o[r][2];
            ws[(h0 + 1) * kOStride + d + 8] = s.o[r][3];
        }
        if (lane < 4) {
            wm[h0] = s.m0;
            wm[h0 + 1] = s.m1;
            wm[8 + h0] = s.l0;
            wm[8 + h0 + 1] = s.l1;
        }
    }
    __syncthreads();

    // Merge the accumulators in order; a thread handles (head, 4 dims), so a
    // warp reads one head's row of each state as 32 consecutive float4.
    auto acc_base = [&](int v) {
        return reinterpret_cast<const float *>(smem + (v % kWarps) * kStages * kTileBytes) +
               (v / kWarps) * kAccFloats;
    };
    const int64_t row_base = static_cast<int64_t>(lb) * sh.Hq + g * G;
    for (int e = threadIdx.x; e < G * (kHeadDim / 4); e += blockDim.x) {
        const int h = e / (kHeadDim / 4);
        const int d0 = (e % (kHeadDim / 4)) * 4;
        float M = -INFINITY;
#pragma unroll
        for (int v = 0; v < kAccs; ++v) M = fmaxf(M, acc_base(v)[kMaxGroup * kOStride + h]);
        float lsum = 0.f;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int v = 0; v < kAccs; ++v) {
            const float *wsv = acc_base(v);
            const float *wmv = wsv + kMaxGroup * kOStride;
            const float sc = ex2(wmv[h] - M);      // an accumulator with no tile: m = -inf, 0
            lsum += sc * wmv[8 + h];
            const float4 x = *reinterpret_cast<const float4 *>(wsv + h * kOStride + d0);
            acc.x += sc * x.x;
            acc.y += sc * x.y;
            acc.z += sc * x.z;
            acc.w += sc * x.w;
        }
        if (nsplit == 1) {
            const float inv = 1.f / lsum;
            if (a.out_bf16) {
                uint2 pk;
                float r0, r1;
                pk.x = pack_bf16(acc.x * inv, acc.y * inv, r0, r1);
                pk.y = pack_bf16(acc.z * inv, acc.w * inv, r0, r1);
                *reinterpret_cast<uint2 *>(reinterpret_cast<uint16_t *>(a.out) +
                                           (row_base + h) * kHeadDim + d0) = pk;
            } else {
                *reinterpret_cast<float4 *>(a.out + (row_base + h) * kHeadDim + d0) =
                    make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
            }
        } else {
            const int64_t prow = (row_base + h) * a.max_splits + split;
            *reinterpret_cast<float4 *>(a.part_o + prow * kHeadDim + d0) = acc;
            if (d0 == 0) {
                a.part_ml[prow * 2] = M;
                a.part_ml[prow * 2 + 1] = lsum;
            }
        }
    }
    if (nsplit == 1 || nsplit > a.merge_max_splits) return;

    // Arrival. Every split of the group arrives once, whatever happened in
    // it; the last one merges the group's G heads (a warp per head) and
    // resets the counter for the next call, which touches it only after this
    // grid has completed.
    __shared__ int s_last;
    __syncthreads();
    if (threadIdx.x == 0) {
        int32_t *counter = a.counters + static_cast<int64_t>(lb) * sh.Hkv + g;
        const bool last = arrive(counter) == nsplit - 1;
        if (last) *counter = 0;
        s_last = last;
    }
    __syncthreads();
    if (!s_last) return;
#pragma unroll 1
    for (int h = warp; h < G; h += kWarps) merge_head_regs(a, row_base + h, nsplit, lane);
}

// K2 for tables of at most kRegMergeMax splits: one warp per (layer-batch
// row, q-head), four per CTA, folding the four chains side by side from
// registers (merge_head_regs), so no shared memory or CTA barrier sits
// between its loads and its store.
__global__ void __launch_bounds__(128) decode_combine_small_kernel(const DecodeArgs a) {
    asm volatile("griddepcontrol.launch_dependents;");   // a following overlapped call
    const int64_t row = static_cast<int64_t>(blockIdx.x) * 4 + (threadIdx.x >> 5);
    if (row >= static_cast<int64_t>(a.nlayers) * a.B * a.s.Hq) return;
    const int b = static_cast<int>((row / a.s.Hq) % a.B);
    // seq_lens is read before the wait, as K1 reads it (no decode kernel writes it)
    const int T = a.seq_lens[b];
    if (T < 1 || T > a.max_blocks * a.s.bt) return;
    const int ns = num_splits(T);
    if (ns <= 1 || ns <= a.merge_max_splits) return;   // written by K1
    asm volatile("griddepcontrol.wait;" ::: "memory");
    merge_head_regs(a, row, ns, threadIdx.x & 31);
}

// K2 for wider tables: one CTA (4 warps) per (layer-batch row, q-head) of a
// multi-split session the split kernel did not merge. Warp w folds chain w, the contiguous quarter
// [w*ns/4, (w+1)*ns/4) of the splits (split order), then warp 0 merges the
// four chains in order. The result depends only on the partials
// and ns. Launched as a programmatic dependent of K1: it waits for K1's
// completion with griddepcontrol.wait, so its CTAs can already be resident
// while K1 drains.
__global__ void __launch_bounds__(128) decode_combine_kernel(const DecodeArgs a) {
    asm volatile("griddepcontrol.launch_dependents;");   // a following overlapped call
    const int64_t row = blockIdx.x;                // lb * Hq + h
    const int lb = static_cast<int>(row / a.s.Hq);
    const int b = lb % a.B;
    // seq_lens is read before the wait, as K1 reads it: no decode kernel
    // writes it, so only the partials have to wait for K1 to finish.
    const int T = a.seq_lens[b];
    if (T < 1 || T > a.max_blocks * a.s.bt) return;
    const int ns = num_splits(T);
    if (ns <= 1 || ns <= a.merge_max_splits) return;   // written by K1
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t base = row * a.max_splits;
    const float2 *ml = reinterpret_cast<const float2 *>(a.part_ml) + base;
    const float4 *po = reinterpret_cast<const float4 *>(a.part_o + base * kHeadDim) + lane;
    __shared__ float s_m[kCombineWarps], s_l[kCombineWarps];
    __shared__ float4 s_acc[kCombineWarps][kHeadDim / 4];

    const int s0 = (warp * ns) / kCombineWarps;
    const int s1 = ((warp + 1) * ns) / kCombineWarps;
    float m = -INFINITY, lsum = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    // Batches of kCombineBatch splits: every load of a batch is issued before
    // the first is folded (indices clamped into the quarter, no guards).
    constexpr int kCombineBatch = 16;
    for (int sb = s0; sb < s1; sb += kCombineBatch) {
        float2 v[kCombineBatch];
        float4 o[kCombineBatch];
#pragma unroll
        for (int j = 0; j < kCombineBatch; ++j) {
            const int sp = min(sb + j, s1 - 1);
            v[j] = ml[sp];
            o[j] = po[sp * (kHeadDim / 4)];
        }
#pragma unroll
        for (int j = 0; j < kCombineBatch; ++j)
            if (sb + j < s1) lse_step(m, lsum, acc, v[j], o[j]);
    }
    s_acc[warp][lane] = acc;
    if (lane == 0) {
        s_m[warp] = m;
        s_l[warp] = lsum;
    }
    __syncthreads();
    if (warp == 0) {
        float mq[kMergeChains], lq[kMergeChains];
        float4 aq[kMergeChains];
#pragma unroll
        for (int q = 0; q < kMergeChains; ++q) {
            mq[q] = s_m[q];
            lq[q] = s_l[q];
            aq[q] = s_acc[q][lane];
        }
        merge_chains_store(a, row, lane, mq, lq, aq);
    }
}

}  // namespace

bool encode_hot_tensor_map(CUtensorMap *map, void *hot_base, int64_t rows, int64_t run_rows,
                           const char **why) {
    // Resolved once; a function-local static is initialised exactly once even
    // when pools are created, or allocation-free decodes issued, on several
    // host threads at the same moment.
    static const PFN_cuTensorMapEncodeTiled_v12000 encode = [] {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                             cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            fn = nullptr;
        return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }();
    if (!encode) {
        *why = "cuTensorMapEncodeTiled entry point unavailable";
        return false;
    }
    // A 4-D view of the pool: (64 columns, row, column half, K|V) with byte
    // strides (2, 256, 128, run_rows * 256). A tile is one box of it: 16 rows
    // of both halves of K and of V, landing in shared memory as [K|V][half]
    // [row][64] with the 128-byte swizzle, the layout the kernel reads.
    cuuint64_t dims[4] = {64, static_cast<cuuint64_t>(rows), 2, 2};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(kRowBytes), 128,
                             static_cast<cuuint64_t>(run_rows) * kRowBytes};
    cuuint32_t box[4] = {64, kTileTokens, 2, 2};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, hot_base, dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        *why = "cuTensorMapEncodeTiled rejected the hot pool";
        return false;
    }
    return true;
}

cudaError_t prepare_kernels() {
    cudaError_t e = cudaFuncSetAttribute(decode_split_kernel<kWarpsNarrow, kStagesFull>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         decode_smem(kWarpsNarrow, kStagesFull));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(decode_split_kernel<kWarpsNarrow, kStagesHalf>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 decode_smem(kWarpsNarrow, kStagesHalf));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(decode_split_kernel<kWarpsWide, kStagesOne>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 decode_smem(kWarpsWide, kStagesOne));
    return e;
}

cudaError_t launch_decode(const CUtensorMap &map, const DecodeArgs &a, int num_sms,
                          cudaStream_t st, bool overlap_previous) {
    // Every session of the batch has T <= max_blocks * bt, so its splits fit.
    const int splits = max_splits_for(static_cast<int64_t>(a.max_blocks) * a.s.bt);
    if (splits > a.max_splits) return cudaErrorInvalidValue;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;

    cudaLaunchConfig_t c1 = {};
    c1.gridDim = dim3(splits, a.s.Hkv, a.nlayers * a.B);
    c1.blockDim = dim3(kWarpsNarrow * 32);
    c1.stream = st;
    c1.attrs = overlap_previous ? attr : nullptr;
    c1.numAttrs = overlap_previous ? 1 : 0;
    // CTAs of the grid (an upper bound: splits past a session's own count
    // exit at once) against the SMs decide the ring depth.
    const int64_t ctas = static_cast<int64_t>(splits) * a.s.Hkv * a.nlayers * a.B;
    // Beyond two CTAs per SM, 2 per SM still wins when it fills its last wave
    // clearly better than 3 per SM (a grid just above one 3-per-SM wave).
    auto fill = [&](int per_sm) {
        const double w = static_cast<double>(ctas) / (per_sm * static_cast<double>(num_sms));
        return w / static_cast<double>(static_cast<int64_t>(w) + (w > static_cast<int64_t>(w)));
    };
    // Which sessions the split kernel merges itself (the bits are the same
    // either way): those of up to kSplitKernelMerge splits, in grids of at
    // least 8 CTAs per SM. There, many groups finish at different times and
    // their merges spread over the grid. In shorter grids each CTA's arrival
    // (an atomic round trip holding its SM slot) and the tail merges cost more
    // than the combine launch (measured on GB300 against merging everything in
    // the combine: 256 x 4K-token sessions per layer +1.3 %, 8 x 4K all
    // layers +1.6 %; one 4K- or 16K-token session per layer -7 % / -5 % and
    // 32 x 4K -5 % when shorter grids merged too).
    DecodeArgs ka = a;
    ka.merge_max_splits = ctas >= 8 * static_cast<int64_t>(num_sms) ? kSplitKernelMerge : 0;
    cudaError_t e;
    if (ctas <= num_sms) {
        c1.blockDim = dim3(kWarpsWide * 32);
        c1.dynamicSmemBytes = decode_smem(kWarpsWide, kStagesOne);
        e = cudaLaunchKernelEx(&c1, decode_split_kernel<kWarpsWide, kStagesOne>, map, ka);
    } else if (ctas <= 2 * static_cast<int64_t>(num_sms) || fill(2) > fill(3) + KVT_WAVE_MARGIN) {
        c1.dynamicSmemBytes = decode_smem(kWarpsNarrow, kStagesHalf);
        e = cudaLaunchKernelEx(&c1, decode_split_kernel<kWarpsNarrow, kStagesHalf>, map, ka);
    } else {
        c1.dynamicSmemBytes = decode_smem(kWarpsNarrow, kStagesFull);
        e = cudaLaunchKernelEx(&c1, decode_split_kernel<kWarpsNarrow, kStagesFull>, map, ka);
    }
    if (e != cudaSuccess) return e;
    // Every session's output written by the split kernel: one split each, or
    // few enough splits to merge there.
    if (splits <= 1 || splits <= ka.merge_max_splits) return cudaSuccess;

    const int64_t rows = static_cast<int64_t>(a.nlayers) * a.B * a.s.Hq;
    cudaLaunchConfig_t c2 = {};
    c2.blockDim = dim3(kCombineWarps * 32);
    c2.dynamicSmemBytes = 0;
    c2.stream = st;
    c2.attrs = attr;
    c2.numAttrs = 1;
    if (splits <= kRegMergeMax) {
        c2.gridDim = dim3(static_cast<unsigned>((rows + 3) / 4));
        return cudaLaunchKernelEx(&c2, decode_combine_small_kernel, ka);
    }
    c2.gridDim = dim3(static_cast<unsigned>(rows));
    return cudaLaunchKernelEx(&c2, decode_combine_kernel, ka);
}

}  // namespace kvt
