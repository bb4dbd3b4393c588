// decode_attention_noalloc: the decode-attention path for callers that must
// not allocate device memory (see include/kvtier.h).
//
// The split-KV decode keeps per-split partial results (running max, sum and
// an unnormalised 128-float accumulator per split and query head) between
// its two kernels. The pool-based entry point keeps them in a workspace the
// pool allocated when it was created; this entry point keeps them in the
// file-scope device array below instead, so a call makes no allocation at
// all. Every GPU that loads the library reserves the array until the
// process exits.
#include <mutex>

#include "../../include/kvtier.h"
#include "kvt_internal.h"

namespace {

constexpr int kMaxDevices = 64;

// Partials (fp32 accumulators, then (max, sum) pairs), then one flag word.
static __device__ __align__(256) unsigned char g_decode_scratch[KV_NOALLOC_SCRATCH_BYTES];
// Split-arrival counters, one per (layer-batch row, kv-head): zero when the
// module loads, and every call leaves them at zero (the last arrival of a
// group resets its counter). They sit apart from the scratch because the
// partials' extent moves with each call's shape and the counters must not.
constexpr int kMaxCounters = 65535 * 8;   // rows x kv-heads at most
static __device__ int32_t g_decode_counters[kMaxCounters];

// Tensor maps of the hot arenas a device's calls have used, so that a call
// over an arena seen before skips the encode (a driver call per decode).
constexpr int kMapCache = 4;
struct CachedMap {
    const void *base = nullptr;
    int64_t rows = 0, run_rows = 0;
    uint64_t last_use = 0;
    CUtensorMap map{};
};

struct DeviceScratch {
    unsigned char *ptr = nullptr;   // device address of g_decode_scratch
    int32_t *counters = nullptr;    // device address of g_decode_counters
    int num_sms = 1;
    bool ready = false;
    CachedMap maps[kMapCache];
    uint64_t clock = 0;
};
DeviceScratch g_dev[kMaxDevices];
std::mutex g_mu;

int fail(int code, const char *msg) {
    kvt::set_last_error(msg);
    return code;
}

// Per-device set-up, run by the first call on each device with that device
// current: the array's device address (the host-side symbol is only a
// stand-in), the decode kernels' shared-memory attributes and the SM count.
int setup_device(int dev, unsigned char **ptr, int32_t **counters, int *num_sms) {
    std::lock_guard<std::mutex> lk(g_mu);
    DeviceScratch &d = g_dev[dev];
    if (!d.ready) {
        void *p = nullptr, *pc = nullptr;
        if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || !p ||
            cudaGetSymbolAddress(&pc, g_decode_counters) != cudaSuccess || !pc)
            return fail(KV_ERR_CUDA, "decode_attention_noalloc: cudaGetSymbolAddress failed");
        if (kvt::prepare_kernels() != cudaSuccess)
            return fail(KV_ERR_CUDA, "decode_attention_noalloc: kernel attribute set-up failed");
        if (cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            return fail(KV_ERR_CUDA, "decode_attention_noalloc: SM count query failed");
        d.ptr = static_cast<unsigned char *>(p);
        d.counters = static_cast<int32_t *>(pc);
        d.ready = true;
    }
    *ptr = d.ptr;
    *counters = d.counters;
    *num_sms = d.num_sms;
    return KV_OK;
}

// The hot arena's tensor map for this device: from the cache, else encoded
// and put in place of the least recently used entry.
int device_tensor_map(int dev, void *hot_base, int64_t rows, int64_t run_rows, CUtensorMap *out) {
    std::lock_guard<std::mutex> lk(g_mu);
    DeviceScratch &d = g_dev[dev];
    CachedMap *victim = &d.maps[0];
    for (CachedMap &m : d.maps) {
        if (m.base == hot_base && m.rows == rows && m.run_rows == run_rows) {
            m.last_use = ++d.clock;
            *out = m.map;
            return KV_OK;
        }
        if (m.last_use < victim->last_use) victim = &m;
    }
    const char *why = nullptr;
    CUtensorMap map;
    if (!kvt::encode_hot_tensor_map(&map, hot_base, rows, run_rows, &why)) return fail(KV_ERR_CUDA, why);
    victim->base = hot_base;
    victim->rows = rows;
    victim->run_rows = run_rows;
    victim->map = map;
    victim->last_use = ++d.clock;
    *out = map;
    return KV_OK;
}

}  // namespace

extern "C" int decode_attention_noalloc(const kv_pool_config *cfg, int32_t layer, const void *q,
                                        const int32_t *block_tables, const int32_t *seq_lens,
                                        int32_t B, int32_t max_blocks, float scale, float *out,
                                        kv_stream_t stream) {
    if (!cfg || !q || !block_tables || !seq_lens || !out || !cfg->hot_base)
        return fail(KV_ERR_INVALID_ARG, "decode_attention_noalloc: null pointer");
    if (((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(block_tables) |
          reinterpret_cast<uintptr_t>(seq_lens)) & 3) || (reinterpret_cast<uintptr_t>(out) & 15))
        return fail(KV_ERR_INVALID_ARG,
                    "decode_attention_noalloc: q, block_tables, seq_lens need 4-byte and out "
                    "16-byte alignment");
    const kv_pool_config &c = *cfg;
    const int G = c.num_kv_heads > 0 ? c.num_q_heads / c.num_kv_heads : 0;
    if (c.head_dim != kvt::kHeadDim || (c.block_tokens != 16 && c.block_tokens != 64) ||
        c.num_kv_heads < 1 || c.num_kv_heads > 8 || c.num_q_heads % c.num_kv_heads != 0 ||
        G < 1 || G > kvt::kMaxGroup || (G & (G - 1)) || c.num_layers < 1 || c.num_hot_blocks < 1)
        return fail(KV_ERR_INVALID_ARG, "decode_attention_noalloc: unsupported shape");
    if (reinterpret_cast<uintptr_t>(c.hot_base) & 255)
        return fail(KV_ERR_INVALID_ARG, "decode_attention_noalloc: hot arena not 256-byte aligned");
    const int64_t rows = c.num_hot_blocks * c.num_layers * 2 * c.num_kv_heads * c.block_tokens;
    if (rows >= (int64_t(1) << 31))
        return fail(KV_ERR_INVALID_ARG, "decode_attention_noalloc: hot pool too large");
    if (layer < -1 || layer >= c.num_layers)
        return fail(KV_ERR_INVALID_ARG, "decode_attention_noalloc: bad layer");
    const int nl = layer < 0 ? c.num_layers : 1;
    if (B < 1 || static_cast<int64_t>(nl) * B > 65535 || max_blocks < 1 || max_blocks > (1 << 26))
        return fail(KV_ERR_INVALID_ARG, "decode_attention_noalloc: B or max_blocks out of range");
    if (!(scale == scale) || scale > 3.0e38f || scale < -3.0e38f)
        return fail(KV_ERR_INVALID_ARG, "decode_attention_noalloc: scale not finite");

    const int splits = kvt::max_splits_for(static_cast<int64_t>(max_blocks) * c.block_tokens);
    const int64_t prow = static_cast<int64_t>(nl) * B * c.num_q_heads * splits;
    const int64_t o_bytes = prow * kvt::kHeadDim * 4;
    const int64_t ml_bytes = prow * 2 * 4;
    if (o_bytes + ml_bytes + 256 > KV_NOALLOC_SCRATCH_BYTES)
        return fail(KV_ERR_INVALID_ARG,
                    "decode_attention_noalloc: batch needs more scratch than the fixed "
                    "KV_NOALLOC_SCRATCH_BYTES; use decode_attention with a pool, or fewer "
                    "sessions / shorter max_blocks per call");

    int prev = -1;
    if (cudaGetDevice(&prev) != cudaSuccess) return fail(KV_ERR_CUDA, "cudaGetDevice failed");
    if (c.device < 0 || c.device >= kMaxDevices)
        return fail(KV_ERR_INVALID_ARG, "decode_attention_noalloc: bad device ordinal");
    if (prev != c.device && cudaSetDevice(c.device) != cudaSuccess)
        return fail(KV_ERR_CUDA, "cudaSetDevice failed");
    struct Restore {
        int dev, cur;
        ~Restore() {
            if (dev >= 0 && dev != cur) cudaSetDevice(dev);
        }
    } restore{prev, c.device};

    unsigned char *scratch = nullptr;
    int32_t *counters = nullptr;
    int num_sms = 1;
    int rc = setup_device(c.device, &scratch, &counters, &num_sms);
    if (rc) return rc;
    CUtensorMap map;
    rc = device_tensor_map(c.device, c.hot_base, rows,
                           static_cast<int64_t>(c.num_kv_heads) * c.block_tokens, &map);
    if (rc) return rc;

    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    // The kernels OR their bounds-check bits into this word. Nothing reads it
    // (this entry point has no pool to report through), so it needs no
    // clearing; no other scratch has to start at zero, since every partial
    // is written before it is read within the call.
    int32_t *flag = reinterpret_cast<int32_t *>(scratch + KV_NOALLOC_SCRATCH_BYTES - 256);

    kvt::DecodeArgs a;
    a.q = static_cast<const uint16_t *>(q);
    a.tables = block_tables;
    a.seq_lens = seq_lens;
    a.out = out;
    a.part_o = reinterpret_cast<float *>(scratch);
    a.part_ml = reinterpret_cast<float *>(scratch + o_bytes);
    a.counters = counters;
    a.err = flag;
    a.B = B;
    a.max_blocks = max_blocks;
    a.layer0 = layer < 0 ? 0 : layer;
    a.nlayers = nl;
    a.max_splits = splits;
    a.scale_log2 = scale * 1.4426950408889634f;
    a.out_bf16 = 0;
    a.k_new = a.v_new = nullptr;
    a.hot = nullptr;
    a.inject_extra_tx = 0;
    a.s = kvt::Shape{c.num_layers, c.num_q_heads, c.num_kv_heads, c.block_tokens, c.num_hot_blocks};
    if (kvt::launch_decode(map, a, num_sms, st, false) != cudaSuccess)
        return fail(KV_ERR_CUDA, "decode_attention_noalloc: kernel launch failed");
    return KV_OK;
}
