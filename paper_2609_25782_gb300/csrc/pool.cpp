// Pool runtime behind the C ABI of include/kvtier.h.
//
// Owns the host metadata of the hot-cold KV hierarchy (Section 3 of the
// paper): the hot free list and per-session block tables, the cold-arena
// placement of per-session images, the session states {ACTIVE, PAUSED}, the
// write-on-evict watermark (cold_valid), and the CUDA events that order
// migrations against decode. Device work goes to the kernels in
// decode_kernels.cu and copy_kernels.cu.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <map>
#include <set>
#include <string>
#include <vector>

#include "../../include/kvtier.h"
#include "kvt_internal.h"

static_assert(KV_DEVICE_BAD_BLOCK == kvt::kErrBadBlock && KV_DEVICE_BAD_LENGTH == kvt::kErrBadLength &&
                  KV_DEVICE_TIMEOUT == kvt::kErrTimeout,
              "public device flag bits must match the kernels'");

namespace {

thread_local std::string g_last_error;

int fail(int code, const std::string &msg) {
    g_last_error = msg;
    return code;
}

// splitmix64 (Steele, Lea, Flood 2014): state += golden gamma, then mix.
uint64_t splitmix64(uint64_t &st) {
    uint64_t z = (st += 0x9E3779B97F4A7C15ULL);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

// Fisher-Yates from the top; draw j = floor(r * (i+1) / 2^64).
void fisher_yates(std::vector<int32_t> &v, size_t n, uint64_t seed) {
    uint64_t st = seed;
    for (size_t i = n; i-- > 1;) {
        const uint64_t r = splitmix64(st);
        const size_t j = static_cast<size_t>((static_cast<unsigned __int128>(r) * (i + 1)) >> 64);
        std::swap(v[i], v[j]);
    }
}

struct Session {
    int32_t state = KV_SESSION_FREE;
    int64_t T = 0, cap = 0, cold_valid = 0;
    int64_t img_off = -1, img_bytes = 0;
    std::vector<int32_t> blocks;      // per logical block: hot slot, or -1 (residency mode)
    std::vector<int16_t> img_tok;     // residency mode: tokens of block j held by the image
    int64_t hot_count = 0;            // residency mode: blocks with a hot slot
    uint64_t last_use = 0;            // residency mode: recency stamp
    cudaEvent_t ready = nullptr;
    bool ready_recorded = false;
    cudaEvent_t appended = nullptr;
    bool appended_recorded = false;
    cudaEvent_t packed = nullptr;     // residency mode: after the last eviction that wrote
    bool packed_recorded = false;     // the image (it covers every earlier one)
    int16_t pack_fence = -1;          // simple mode: fence slot and generation of the
    uint64_t pack_gen = 0;            // last pause's pack (it reads the table row)
};

// A planned eviction: block j of session sid leaves hot slot `slot`; tokens
// [t0, t1) are written to the image first (t0 == t1: the image has them).
struct Victim {
    int32_t sid, j, slot, t0, t1;
};

constexpr int kFenceSlots = 64;
struct Fence {
    cudaEvent_t ev = nullptr;
    uint64_t gen = 0;
};

class DeviceGuard {
  public:
    DeviceGuard(int dev, bool active) : active_(active) {
        if (active_ && cudaGetDevice(&prev_) == cudaSuccess && prev_ != dev) cudaSetDevice(dev);
        else prev_ = -1;
    }
    ~DeviceGuard() {
        if (active_ && prev_ >= 0) cudaSetDevice(prev_);
    }

  private:
    bool active_;
    int prev_ = -1;
};

}  // namespace

void kvt::set_last_error(const char *msg) { g_last_error = msg; }

struct kv_pool {
    kv_pool_config cfg{};
    bool host_only = false;
    int64_t block_bytes = 0, token_bytes = 0;
    int32_t table_stride = 0;            // max blocks per session
    int32_t max_splits = 0;              // split bound for max_context
    int64_t part_rows = 0;               // decode workspace capacity (partial rows)
    int num_sms = 1;
    int mig_ctas = 0;                    // cap on migration-kernel CTAs, 0 = none
    kvt::Shape shape{};

    std::vector<int32_t> free_list;      // top = back
    std::vector<int16_t> block_fence;    // fence slot of the pack that freed it, or -1
    std::vector<uint64_t> block_fence_gen;
    std::vector<Session> sessions;
    std::map<int64_t, int64_t> cold_free;  // offset -> bytes
    int64_t cold_used = 0;

    int32_t *d_tables = nullptr;
    float *d_part_o = nullptr;
    float *d_part_ml = nullptr;
    int32_t *d_counters = nullptr;       // split arrivals per (layer-batch row, kv-head)
    int64_t counter_count = 0;
    int32_t *d_err = nullptr;
    CUtensorMap tmap{};

    Fence fences[kFenceSlots];
    int next_fence = 0;
    uint64_t fence_gen = 0;

    kv_pool_stats stats{};
    int32_t inject_countdown = 0;
    bool inject_timeout = false;   // kv_pool_inject_decode_timeout, next decode only

    // Residency mode (KV_POOL_LRU_RESIDENCY): sessions holding hot blocks,
    // ordered by (last use, sid); the first one is the least recently used.
    bool lru = false;
    uint64_t clock = 0;
    std::set<std::pair<uint64_t, int32_t>> lru_set;

    // Every CUDA call of the pool goes through here: the failure-injection
    // hook fires first, then (unless the pool is host-logic only) the call.
    template <typename F>
    int cuda(const char *what, F &&fn) {
        if (inject_countdown > 0 && --inject_countdown == 0)
            return fail(KV_ERR_CUDA, std::string(what) + ": injected CUDA failure");
        if (host_only) return KV_OK;
        cudaError_t e = fn();
        if (e != cudaSuccess)
            return fail(KV_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
        return KV_OK;
    }

    Session *session(int32_t sid) {
        if (sid < 0 || sid >= static_cast<int32_t>(sessions.size())) return nullptr;
        Session &s = sessions[sid];
        return s.state == KV_SESSION_FREE ? nullptr : &s;
    }

    int64_t image_bytes(int64_t cap) const {
        return (cap * token_bytes + 255) / 256 * 256;
    }

    bool cold_alloc(int64_t bytes, int64_t *off) {
        for (auto it = cold_free.begin(); it != cold_free.end(); ++it) {
            if (it->second >= bytes) {
                *off = it->first;
                const int64_t rest = it->second - bytes;
                const int64_t at = it->first + bytes;
                cold_free.erase(it);
                if (rest > 0) cold_free[at] = rest;
                cold_used += bytes;
                return true;
            }
        }
        return false;
    }

    void cold_release(int64_t off, int64_t bytes) {
        cold_used -= bytes;
        auto it = cold_free.emplace(off, bytes).first;
        auto nx = std::next(it);
        if (nx != cold_free.end() && it->first + it->second == nx->first) {
            it->second += nx->second;
            cold_free.erase(nx);
        }
        if (it != cold_free.begin()) {
            auto pv = std::prev(it);
            if (pv->first + pv->second == it->first) {
                pv->second += it->second;
                cold_free.erase(it);
            }
        }
    }

    // Blocks popped for a session: make `st` wait for the packs that freed
    // them, if those packs may still be running.
    int wait_fences(const int32_t *blocks, size_t n, cudaStream_t st) {
        bool need[kFenceSlots] = {};
        for (size_t i = 0; i < n; ++i) {
            const int f = block_fence[blocks[i]];
            if (f >= 0 && fences[f].gen == block_fence_gen[blocks[i]]) need[f] = true;
        }
        for (int f = 0; f < kFenceSlots; ++f) {
            if (!need[f]) continue;
            int rc = cuda("cudaStreamWaitEvent", [&] { return cudaStreamWaitEvent(st, fences[f].ev, 0); });
            if (rc) return rc;
        }
        return KV_OK;
    }

    void clear_fences(const int32_t *blocks, size_t n) {
        for (size_t i = 0; i < n; ++i) block_fence[blocks[i]] = -1;
    }

    // Write entries [from, from+n) of a session's device table row.
    int write_table(int32_t sid, const int32_t *vals, int64_t from, int64_t n, cudaStream_t st) {
        for (int64_t i = 0; i < n; i += kvt::kTableWriteMax) {
            kvt::TableWriteArgs a;
            a.dst = d_tables + static_cast<int64_t>(sid) * table_stride + from + i;
            a.n = static_cast<int32_t>(std::min<int64_t>(kvt::kTableWriteMax, n - i));
            std::memcpy(a.vals, vals + i, sizeof(int32_t) * a.n);
            int rc = cuda("table write launch", [&] { return kvt::launch_table_write(a, st); });
            if (rc) return rc;
        }
        return KV_OK;
    }

    // ---- residency mode -------------------------------------------------
    int32_t tokens_in_block(const Session &s, int64_t j) const {
        const int64_t n = s.T - j * cfg.block_tokens;
        return static_cast<int32_t>(n < cfg.block_tokens ? n : cfg.block_tokens);
    }

    void lru_out(int32_t sid) {
        Session &s = sessions[sid];
        if (s.hot_count > 0) lru_set.erase({s.last_use, sid});
    }
    void lru_in(int32_t sid) {
        Session &s = sessions[sid];
        if (s.hot_count > 0) lru_set.insert({s.last_use, sid});
    }

    // Least recently used hot blocks, outside `protect`, until `need` blocks
    // would be free. Sessions in recency order; within one, ascending j.
    bool plan_evict(int64_t need, const std::vector<int32_t> &protect, std::vector<Victim> &out) {
        int64_t have = static_cast<int64_t>(free_list.size());
        for (const auto &e : lru_set) {
            if (have >= need) break;
            const int32_t sid = e.second;
            if (std::find(protect.begin(), protect.end(), sid) != protect.end()) continue;
            const Session &s = sessions[sid];
            for (size_t j = 0; j < s.blocks.size() && have < need; ++j) {
                if (s.blocks[j] < 0) continue;
                out.push_back({sid, static_cast<int32_t>(j), s.blocks[j], s.img_tok[j],
                               tokens_in_block(s, static_cast<int64_t>(j))});
                ++have;
            }
        }
        return have >= need;
    }

    // The `need` slots the call will pop once the victims are pushed back:
    // the free list grows by the victims (in order), pops come off its end.
    std::vector<int32_t> peek_alloc(int64_t need, const std::vector<Victim> &v) const {
        std::vector<int32_t> all(free_list);
        for (const Victim &x : v) all.push_back(x.slot);
        std::vector<int32_t> out(need);
        for (int64_t i = 0; i < need; ++i) out[i] = all[all.size() - 1 - i];
        return out;
    }

    // Device side of the victims: wait for their last writes, then write the
    // tokens each image lacks. A session whose image this writes records its
    // `packed` event after the writes; the stream first waits for the previous
    // recording, so the event covers every eviction of the session so far.
    // Whatever later fetches the session's blocks back waits on it
    // (wait_packed), on whichever stream it runs.
    int evict_device(const std::vector<Victim> &v, cudaStream_t st) {
        std::vector<int32_t> seen, writes;
        for (const Victim &x : v) {
            if (x.t1 > x.t0 && std::find(writes.begin(), writes.end(), x.sid) == writes.end())
                writes.push_back(x.sid);
            if (std::find(seen.begin(), seen.end(), x.sid) != seen.end()) continue;
            seen.push_back(x.sid);
            Session &s = sessions[x.sid];
            int rc = KV_OK;
            if (s.appended_recorded)
                rc = cuda("cudaStreamWaitEvent", [&] { return cudaStreamWaitEvent(st, s.appended, 0); });
            if (!rc && s.ready_recorded)
                rc = cuda("cudaStreamWaitEvent", [&] { return cudaStreamWaitEvent(st, s.ready, 0); });
            if (!rc) rc = wait_packed(x.sid, st);
            if (rc) return rc;
        }
        std::vector<kvt::BlockJob> jobs;
        for (const Victim &x : v)
            if (x.t1 > x.t0) jobs.push_back(job_for(x.sid, x.j, x.slot, x.t0, x.t1));
        int rc = run_jobs(jobs, true, st);
        for (size_t i = 0; !rc && !host_only && i < writes.size(); ++i) {
            Session &s = sessions[writes[i]];
            if (!s.packed)
                rc = cuda("cudaEventCreate",
                          [&] { return cudaEventCreateWithFlags(&s.packed, cudaEventDisableTiming); });
            if (!rc) rc = cuda("cudaEventRecord", [&] { return cudaEventRecord(s.packed, st); });
        }
        if (rc) return rc;
        for (int32_t sid : writes) sessions[sid].packed_recorded = !host_only;
        return KV_OK;
    }

    // Before blocks of `sid` are fetched from its image on `st`: the image
    // writes of its evictions (possibly on another stream) must be complete.
    int wait_packed(int32_t sid, cudaStream_t st) {
        const Session &s = sessions[sid];
        if (!s.packed_recorded) return KV_OK;
        return cuda("cudaStreamWaitEvent", [&] { return cudaStreamWaitEvent(st, s.packed, 0); });
    }

    void evict_commit(const std::vector<Victim> &v) {
        for (const Victim &x : v) {
            Session &s = sessions[x.sid];
            lru_out(x.sid);
            if (x.t1 > x.t0) stats.bytes_packed += static_cast<int64_t>(x.t1 - x.t0) * token_bytes;
            s.img_tok[x.j] = static_cast<int16_t>(x.t1);
            s.blocks[x.j] = -1;
            s.hot_count -= 1;
            lru_in(x.sid);
            free_list.push_back(x.slot);
            stats.blocks_evicted += 1;
            stats.free_blocks += 1;
            stats.used_blocks -= 1;
        }
    }

    kvt::BlockJob job_for(int32_t sid, int32_t j, int32_t slot, int32_t t0, int32_t t1) const {
        const Session &s = sessions[sid];
        kvt::BlockJob b;
        b.img = static_cast<uint8_t *>(cfg.cold_base) + s.img_off;
        b.T_cap = static_cast<int32_t>(s.cap);
        b.sid = -1;
        b.slot = slot;
        b.j = j;
        b.t0 = t0;
        b.t1 = t1;
        return b;
    }

    // A fetch of block j into `slot`: the copy also writes the session's
    // device table entry j.
    kvt::BlockJob fetch_job(int32_t sid, int32_t j, int32_t slot, int32_t t0, int32_t t1) const {
        kvt::BlockJob b = job_for(sid, j, slot, t0, t1);
        b.sid = sid;
        return b;
    }

    int run_jobs(const std::vector<kvt::BlockJob> &jobs, bool pack, cudaStream_t st) {
        for (size_t i = 0; i < jobs.size(); i += kvt::kBlockJobsMax) {
            kvt::BlockJobs a;
            a.hot = static_cast<uint8_t *>(cfg.hot_base);
            a.err = d_err;
            a.tables = d_tables;
            a.table_stride = table_stride;
            a.s = shape;
            a.n = static_cast<int32_t>(std::min<size_t>(kvt::kBlockJobsMax, jobs.size() - i));
            a.pad = 0;
            std::copy(jobs.begin() + i, jobs.begin() + i + a.n, a.job);
            int rc = cuda(pack ? "pack launch" : "unpack launch",
                          [&] { return kvt::launch_block_jobs(a, pack, num_sms, mig_ctas, st); });
            if (rc) return rc;
        }
        return KV_OK;
    }

    kvt::MigArgs mig_args(int32_t sid, const Session &s) const {
        kvt::MigArgs m;
        m.table = d_tables + static_cast<int64_t>(sid) * table_stride;
        m.hot = static_cast<uint8_t *>(cfg.hot_base);
        m.img = static_cast<uint8_t *>(cfg.cold_base) + s.img_off;
        m.T_cap = s.cap;
        m.t_begin = 0;
        m.t_end = 0;
        m.err = d_err;
        m.s = shape;
        return m;
    }
};

extern "C" {

const char *kv_last_error(void) { return g_last_error.c_str(); }

int64_t kv_token_bytes(const kv_pool_config *c) {
    return c ? static_cast<int64_t>(c->num_layers) * 2 * c->num_kv_heads * c->head_dim * 2 : 0;
}

int64_t kv_block_bytes(const kv_pool_config *c) {
    return c ? kv_token_bytes(c) * c->block_tokens : 0;
}

int32_t kv_decode_splits(int64_t t) {
    return t < 1 ? 0 : kvt::max_splits_for(t);
}

int kv_pool_create(const kv_pool_config *cfg, kv_pool **out) {
    if (!cfg || !out) return fail(KV_ERR_INVALID_ARG, "kv_pool_create: null argument");
    const kv_pool_config &c = *cfg;
    if (c.head_dim != kvt::kHeadDim) return fail(KV_ERR_INVALID_ARG, "head_dim must be 128");
    if (c.block_tokens != 16 && c.block_tokens != 64)
        return fail(KV_ERR_INVALID_ARG, "block_tokens must be 16 or 64");
    if (c.num_layers < 1 || c.num_kv_heads < 1 || c.num_kv_heads > 8 || c.num_q_heads < 1 ||
        c.num_q_heads % c.num_kv_heads != 0 || c.num_q_heads / c.num_kv_heads > kvt::kMaxGroup ||
        (c.num_q_heads / c.num_kv_heads) & (c.num_q_heads / c.num_kv_heads - 1))
        return fail(KV_ERR_INVALID_ARG, "need Hkv in 1..8 and Hq/Hkv in {1,2,4,8}");
    if (c.max_sessions < 1 || c.max_batch < 1 || c.max_context < 1 || c.num_hot_blocks < 1)
        return fail(KV_ERR_INVALID_ARG, "max_sessions, max_batch, max_context, num_hot_blocks must be >= 1");
    if (c.num_hot_blocks > INT32_MAX)
        return fail(KV_ERR_INVALID_ARG, "num_hot_blocks exceeds int32 block ids");
    const int64_t rows = c.num_hot_blocks * c.num_layers * 2 * c.num_kv_heads * c.block_tokens;
    if (rows >= (int64_t(1) << 31))
        return fail(KV_ERR_INVALID_ARG, "hot pool has 2^31 or more 256-byte rows");
    if (c.max_context > (int64_t(1) << 30)) return fail(KV_ERR_INVALID_ARG, "max_context too large");
    const bool host_only = (c.flags & KV_POOL_HOST_LOGIC_ONLY) != 0;
    if (!host_only) {
        if (!c.hot_base || !c.cold_base) return fail(KV_ERR_INVALID_ARG, "null arena");
        if ((reinterpret_cast<uintptr_t>(c.hot_base) & 255) ||
            (reinterpret_cast<uintptr_t>(c.cold_base) & 255))
            return fail(KV_ERR_INVALID_ARG, "arenas must be 256-byte aligned");
    }
    if (c.cold_bytes < 0) return fail(KV_ERR_INVALID_ARG, "cold_bytes < 0");

    kv_pool *p = new kv_pool;
    p->cfg = c;
    p->host_only = host_only;
    p->lru = (c.flags & KV_POOL_LRU_RESIDENCY) != 0;
    p->token_bytes = kv_token_bytes(&c);
    p->block_bytes = kv_block_bytes(&c);
    p->table_stride = static_cast<int32_t>((c.max_context + c.block_tokens - 1) / c.block_tokens);
    p->max_splits = kvt::max_splits_for(static_cast<int64_t>(p->table_stride) * c.block_tokens);
    p->shape = kvt::Shape{c.num_layers, c.num_q_heads, c.num_kv_heads, c.block_tokens,
                          c.num_hot_blocks};
    p->free_list.resize(c.num_hot_blocks);
    for (int64_t i = 0; i < c.num_hot_blocks; ++i) p->free_list[i] = static_cast<int32_t>(i);
    fisher_yates(p->free_list, p->free_list.size(), c.alloc_seed);
    p->block_fence.assign(c.num_hot_blocks, -1);
    p->block_fence_gen.assign(c.num_hot_blocks, 0);
    p->sessions.resize(c.max_sessions);
    if (c.cold_bytes > 0) p->cold_free[0] = c.cold_bytes;

    // decode workspace capacity (also checked against calls on host-logic pools)
    p->part_rows = static_cast<int64_t>(c.max_batch) * c.num_q_heads * p->max_splits;
    if (!host_only) {
        DeviceGuard dg(c.device, true);
        auto bail = [&](int rc) {
            kv_pool_destroy(p);
            return rc;
        };
        if (cudaSetDevice(c.device) != cudaSuccess)
            return bail(fail(KV_ERR_CUDA, "cudaSetDevice failed"));
        cudaDeviceGetAttribute(&p->num_sms, cudaDevAttrMultiProcessorCount, c.device);
        const int64_t tbl = static_cast<int64_t>(c.max_sessions) * p->table_stride * 4;
        const int64_t prow = p->part_rows;
        int rc = p->cuda("cudaMalloc(tables)", [&] { return cudaMalloc(&p->d_tables, tbl); });
        if (!rc) rc = p->cuda("cudaMalloc(partials)", [&] {
            return cudaMalloc(&p->d_part_o, prow * kvt::kHeadDim * sizeof(float));
        });
        if (!rc) rc = p->cuda("cudaMalloc(partials)", [&] {
            return cudaMalloc(&p->d_part_ml, prow * 2 * sizeof(float));
        });
        // A multi-split call has at most part_rows / Hq layer-batch rows.
        p->counter_count = prow / c.num_q_heads * c.num_kv_heads;
        const int64_t cnt = p->counter_count * 4;
        if (!rc) rc = p->cuda("cudaMalloc(counters)", [&] { return cudaMalloc(&p->d_counters, cnt); });
        if (!rc) rc = p->cuda("cudaMemset", [&] { return cudaMemset(p->d_counters, 0, cnt); });
        if (!rc) rc = p->cuda("cudaMalloc(err)", [&] { return cudaMalloc(&p->d_err, 4); });
        if (!rc) rc = p->cuda("cudaMemset", [&] { return cudaMemset(p->d_err, 0, 4); });
        if (!rc) rc = p->cuda("cudaMemset", [&] { return cudaMemset(p->d_tables, 0xFF, tbl); });
        if (!rc) rc = p->cuda("kernel attributes", [&] { return kvt::prepare_kernels(); });
        for (int f = 0; !rc && f < kFenceSlots; ++f)
            rc = p->cuda("cudaEventCreate", [&] {
                return cudaEventCreateWithFlags(&p->fences[f].ev, cudaEventDisableTiming);
            });
        if (rc) return bail(rc);
        const char *why = nullptr;
        if (!kvt::encode_hot_tensor_map(&p->tmap, c.hot_base, rows,
                                        static_cast<int64_t>(c.num_kv_heads) * c.block_tokens, &why))
            return bail(fail(KV_ERR_CUDA, why));
        if (cudaDeviceSynchronize() != cudaSuccess)
            return bail(fail(KV_ERR_CUDA, "device synchronise after pool set-up failed"));
    }
    p->stats.free_blocks = c.num_hot_blocks;
    *out = p;
    return KV_OK;
}

int kv_pool_destroy(kv_pool *p) {
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    if (!p->host_only) {
        DeviceGuard dg(p->cfg.device, true);
        cudaDeviceSynchronize();
        for (auto &s : p->sessions) {
            if (s.ready) cudaEventDestroy(s.ready);
            if (s.appended) cudaEventDestroy(s.appended);
            if (s.packed) cudaEventDestroy(s.packed);
        }
        for (auto &f : p->fences)
            if (f.ev) cudaEventDestroy(f.ev);
        cudaFree(p->d_tables);
        cudaFree(p->d_part_o);
        cudaFree(p->d_part_ml);
        cudaFree(p->d_counters);
        cudaFree(p->d_err);
    }
    delete p;
    return KV_OK;
}

static int create_session(kv_pool *p, int64_t max_tokens, int64_t tokens, int32_t state,
                          int32_t *sid_out) {
    if (!p || !sid_out) return fail(KV_ERR_INVALID_ARG, "null argument");
    if (max_tokens < 1 || max_tokens > p->cfg.max_context)
        return fail(KV_ERR_INVALID_ARG, "max_tokens must be in 1..max_context");
    if (tokens < 0 || tokens > max_tokens) return fail(KV_ERR_INVALID_ARG, "tokens out of range");
    int32_t sid = -1;
    for (int32_t i = 0; i < static_cast<int32_t>(p->sessions.size()); ++i)
        if (p->sessions[i].state == KV_SESSION_FREE) {
            sid = i;
            break;
        }
    if (sid < 0) return fail(KV_ERR_INVALID_ARG, "no free session id (max_sessions reached)");
    const int64_t bytes = p->image_bytes(max_tokens);
    int64_t off = 0;
    if (!p->cold_alloc(bytes, &off))
        return fail(KV_ERR_NO_COLD_SPACE, "cold arena cannot hold the session image");
    Session &s = p->sessions[sid];
    s = Session{};
    s.state = state;
    s.cap = max_tokens;
    s.T = tokens;
    s.cold_valid = tokens;
    s.img_off = off;
    s.img_bytes = bytes;
    if (p->lru && tokens > 0) {   // the image holds every block, none is hot
        const int64_t nb = (tokens + p->cfg.block_tokens - 1) / p->cfg.block_tokens;
        s.blocks.assign(nb, -1);
        s.img_tok.resize(nb);
        for (int64_t j = 0; j < nb; ++j) s.img_tok[j] = static_cast<int16_t>(p->tokens_in_block(s, j));
    }
    p->stats.cold_bytes_used = p->cold_used;
    *sid_out = sid;
    return KV_OK;
}

int session_create(kv_pool *p, int64_t max_tokens, int32_t *sid_out) {
    return create_session(p, max_tokens, 0, KV_SESSION_ACTIVE, sid_out);
}

int session_create_paused(kv_pool *p, int64_t max_tokens, int64_t tokens, int32_t *sid_out) {
    if (tokens < 1) return fail(KV_ERR_INVALID_ARG, "a paused session needs tokens >= 1");
    return create_session(p, max_tokens, tokens, KV_SESSION_PAUSED, sid_out);
}

int session_destroy(kv_pool *p, int32_t sid) {
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    Session *s = p->session(sid);
    if (!s) return fail(KV_ERR_INVALID_ARG, "no such session");
    if (p->lru) p->lru_out(sid);
    int64_t freed = 0;
    for (int32_t b : s->blocks)
        if (b >= 0) {
            p->free_list.push_back(b);
            ++freed;
        }
    p->stats.free_blocks += freed;
    p->stats.used_blocks -= freed;
    p->cold_release(s->img_off, s->img_bytes);
    p->stats.cold_bytes_used = p->cold_used;
    cudaEvent_t ready = s->ready, appended = s->appended, packed = s->packed;
    *s = Session{};
    s->ready = ready;   // events are kept for reuse by the next session in this slot
    s->appended = appended;
    s->packed = packed;
    return KV_OK;
}

// The decode kernels read q as 4-byte words and store out as 16-byte vectors.
static bool decode_pointers_aligned(const void *q, const void *tables, const void *lens,
                                    const void *out) {
    const uintptr_t a4 = reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(tables) |
                         reinterpret_cast<uintptr_t>(lens);
    return (a4 & 3) == 0 && (reinterpret_cast<uintptr_t>(out) & 15) == 0;
}

static int ensure_event(kv_pool *p, cudaEvent_t *ev) {
    if (*ev || p->host_only) return KV_OK;
    return p->cuda("cudaEventCreate",
                   [&] { return cudaEventCreateWithFlags(ev, cudaEventDisableTiming); });
}

// ---- residency mode (KV_POOL_LRU_RESIDENCY) --------------------------------

static int wait_event(kv_pool *p, cudaStream_t st, cudaEvent_t ev) {
    return p->cuda("cudaStreamWaitEvent", [&] { return cudaStreamWaitEvent(st, ev, 0); });
}

// Append with residency: a tail block that was evicted comes back first,
// new blocks come from the free list or from evicting LRU blocks.
static int lru_append(kv_pool *p, int32_t sid, const void *k, const void *v, int32_t n,
                      cudaStream_t st) {
    Session *s = &p->sessions[sid];
    if (s->state != KV_SESSION_ACTIVE) return fail(KV_ERR_BAD_STATE, "append to a paused session");
    if (n < 1) return fail(KV_ERR_INVALID_ARG, "n must be >= 1");
    if (!p->host_only && (!k || !v)) return fail(KV_ERR_INVALID_ARG, "null k or v");
    if ((reinterpret_cast<uintptr_t>(k) | reinterpret_cast<uintptr_t>(v)) & 15)
        return fail(KV_ERR_INVALID_ARG, "k and v must be 16-byte aligned");
    if (s->T + n > s->cap) return fail(KV_ERR_INVALID_ARG, "append past the session capacity");
    const int bt = p->cfg.block_tokens;
    const int64_t have = static_cast<int64_t>(s->blocks.size());
    const int64_t tail = s->T > 0 ? (s->T - 1) / bt : -1;
    const bool refetch = (s->T % bt) != 0 && tail >= 0 && s->blocks[tail] < 0;
    const int64_t fresh_n = (s->T + n + bt - 1) / bt - have;
    const int64_t need = (refetch ? 1 : 0) + fresh_n;
    std::vector<Victim> vic;
    if (!p->plan_evict(need, {sid}, vic))
        return fail(KV_ERR_NO_HOT_BLOCKS, "no block can be evicted for the append");
    const std::vector<int32_t> got = p->peek_alloc(need, vic);

    DeviceGuard dg(p->cfg.device, !p->host_only);
    int rc = ensure_event(p, &s->appended);
    if (!rc && s->ready_recorded) rc = wait_event(p, st, s->ready);
    if (!rc) rc = p->evict_device(vic, st);
    if (!rc && refetch) rc = p->wait_packed(sid, st);
    if (!rc && refetch) {
        rc = p->run_jobs({p->fetch_job(sid, static_cast<int32_t>(tail), got[0], 0,
                                       p->tokens_in_block(*s, tail))}, false, st);
    }
    if (!rc && fresh_n > 0)
        rc = p->write_table(sid, got.data() + (refetch ? 1 : 0), have, fresh_n, st);
    if (!rc) {
        kvt::AppendArgs a;
        a.k = static_cast<const uint8_t *>(k);
        a.v = static_cast<const uint8_t *>(v);
        a.table = p->d_tables + static_cast<int64_t>(sid) * p->table_stride;
        a.hot = static_cast<uint8_t *>(p->cfg.hot_base);
        a.pos0 = s->T;
        a.n = n;
        a.err = p->d_err;
        a.s = p->shape;
        rc = p->cuda("append launch", [&] { return kvt::launch_append(a, p->num_sms, st); });
    }
    if (!rc) rc = p->cuda("cudaEventRecord", [&] { return cudaEventRecord(s->appended, st); });
    if (rc) return rc;   // host state untouched

    p->evict_commit(vic);
    p->free_list.resize(p->free_list.size() - need);
    p->lru_out(sid);
    if (refetch) {
        s->blocks[tail] = got[0];
        s->hot_count += 1;
        p->stats.bytes_unpacked += p->tokens_in_block(*s, tail) * p->token_bytes;
    }
    for (int64_t i = 0; i < fresh_n; ++i) {
        s->blocks.push_back(got[(refetch ? 1 : 0) + i]);
        s->img_tok.push_back(0);
        s->hot_count += 1;
    }
    s->T += n;
    s->last_use = ++p->clock;
    p->lru_in(sid);
    s->appended_recorded = !p->host_only;
    p->stats.free_blocks -= need;
    p->stats.used_blocks += need;
    p->stats.bytes_appended += static_cast<int64_t>(n) * p->token_bytes;
    p->stats.appends += 1;
    return KV_OK;
}

// Resume with residency: only blocks no longer hot are fetched (misses);
// the rest are hits.
static int lru_resume(kv_pool *p, int32_t sid, cudaStream_t st) {
    Session *s = &p->sessions[sid];
    std::vector<int32_t> missing;
    for (size_t j = 0; j < s->blocks.size(); ++j)
        if (s->blocks[j] < 0) missing.push_back(static_cast<int32_t>(j));
    const int64_t need = static_cast<int64_t>(missing.size());
    std::vector<Victim> vic;
    if (!p->plan_evict(need, {sid}, vic))
        return fail(KV_ERR_NO_HOT_BLOCKS, "no block can be evicted for the resume");
    const std::vector<int32_t> got = p->peek_alloc(need, vic);
    std::vector<int32_t> row(s->blocks);
    std::vector<kvt::BlockJob> jobs;
    int64_t fetched = 0;
    for (int64_t i = 0; i < need; ++i) {
        const int32_t j = missing[i];
        row[j] = got[i];
        jobs.push_back(p->fetch_job(sid, j, got[i], 0, p->tokens_in_block(*s, j)));
        fetched += p->tokens_in_block(*s, j);
    }

    DeviceGuard dg(p->cfg.device, !p->host_only);
    int rc = ensure_event(p, &s->ready);
    if (!rc) rc = p->evict_device(vic, st);
    if (!rc && need > 0) rc = p->wait_packed(sid, st);
    if (!rc) rc = p->run_jobs(jobs, false, st);
    if (!rc) rc = p->cuda("cudaEventRecord", [&] { return cudaEventRecord(s->ready, st); });
    if (rc) return rc;

    p->evict_commit(vic);
    p->free_list.resize(p->free_list.size() - need);
    p->lru_out(sid);
    s->blocks = row;
    s->hot_count += need;
    s->state = KV_SESSION_ACTIVE;
    s->last_use = ++p->clock;
    p->lru_in(sid);
    s->ready_recorded = !p->host_only;
    p->stats.free_blocks -= need;
    p->stats.used_blocks += need;
    p->stats.bytes_unpacked += fetched * p->token_bytes;
    p->stats.resume_blocks_hit += static_cast<int64_t>(s->blocks.size()) - need;
    p->stats.resume_blocks_missed += need;
    p->stats.resumes += 1;
    return KV_OK;
}

// Bring back every evicted block of the sessions `uniq` (no pinning: under
// pressure even active blocks spill), with victims from sessions outside
// `protect`, then stamp all of `uniq` with one new recency time. With
// record_ready, each session that had a block fetched re-records its ready
// event on `st` (a decode stream waits on it). *blocks receives the number
// of blocks fetched.
static int lru_fetch(kv_pool *p, const std::vector<int32_t> &uniq,
                     const std::vector<int32_t> &protect, bool record_ready, cudaStream_t st,
                     int64_t *blocks) {
    std::vector<std::vector<int32_t>> miss(uniq.size());
    int64_t need = 0;
    for (size_t u = 0; u < uniq.size(); ++u) {
        const Session &s = p->sessions[uniq[u]];
        for (size_t j = 0; j < s.blocks.size(); ++j)
            if (s.blocks[j] < 0) miss[u].push_back(static_cast<int32_t>(j));
        need += static_cast<int64_t>(miss[u].size());
    }
    std::vector<Victim> vic;
    if (!p->plan_evict(need, protect, vic))
        return fail(KV_ERR_NO_HOT_BLOCKS, "the batch's blocks do not fit in the hot pool");
    const std::vector<int32_t> got = p->peek_alloc(need, vic);
    std::vector<std::vector<int32_t>> rows(uniq.size());
    std::vector<kvt::BlockJob> jobs;
    int64_t k = 0, fetched = 0;
    for (size_t u = 0; u < uniq.size(); ++u) {
        const Session &s = p->sessions[uniq[u]];
        rows[u] = s.blocks;
        for (int32_t j : miss[u]) {
            rows[u][j] = got[k];
            jobs.push_back(p->fetch_job(uniq[u], j, got[k], 0, p->tokens_in_block(s, j)));
            fetched += p->tokens_in_block(s, j);
            ++k;
        }
    }
    int rc = KV_OK;
    for (size_t u = 0; !rc && record_ready && u < uniq.size(); ++u)
        if (!miss[u].empty()) rc = ensure_event(p, &p->sessions[uniq[u]].ready);
    if (!rc) rc = p->evict_device(vic, st);
    for (size_t u = 0; !rc && u < uniq.size(); ++u)
        if (!miss[u].empty()) rc = p->wait_packed(uniq[u], st);
    if (!rc) rc = p->run_jobs(jobs, false, st);   // the fetches also write their table entries
    for (size_t u = 0; !rc && record_ready && !p->host_only && u < uniq.size(); ++u)
        if (!miss[u].empty()) {
            cudaEvent_t ev = p->sessions[uniq[u]].ready;
            rc = p->cuda("cudaEventRecord", [&] { return cudaEventRecord(ev, st); });
        }
    if (rc) return rc;

    p->evict_commit(vic);
    p->free_list.resize(p->free_list.size() - need);
    const uint64_t stamp = ++p->clock;
    for (size_t u = 0; u < uniq.size(); ++u) {
        Session &s = p->sessions[uniq[u]];
        p->lru_out(uniq[u]);
        s.blocks = rows[u];
        s.hot_count += static_cast<int64_t>(miss[u].size());
        s.last_use = stamp;
        p->lru_in(uniq[u]);
        if (record_ready && !miss[u].empty()) s.ready_recorded = !p->host_only;
    }
    p->stats.free_blocks -= need;
    p->stats.used_blocks += need;
    p->stats.bytes_unpacked += fetched * p->token_bytes;
    *blocks = need;
    return KV_OK;
}

static std::vector<int32_t> unique_ids(const int32_t *ids, int32_t n) {
    std::vector<int32_t> u;
    for (int32_t i = 0; i < n; ++i)
        if (std::find(u.begin(), u.end(), ids[i]) == u.end()) u.push_back(ids[i]);
    return u;
}

// Before a decode step: the batch's evicted blocks come back on the step's
// own stream; victims are outside the batch.
static int lru_fetch_batch(kv_pool *p, const int32_t *sids, int32_t B, cudaStream_t st) {
    const std::vector<int32_t> uniq = unique_ids(sids, B);
    int64_t blocks = 0;
    int rc = lru_fetch(p, uniq, uniq, false, st, &blocks);
    if (!rc) p->stats.batch_blocks_fetched += blocks;
    return rc;
}

int session_append(kv_pool *p, int32_t sid, const void *k, const void *v, int32_t n,
                   kv_stream_t stream_) {
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream_);
    Session *s = p->session(sid);
    if (!s) return fail(KV_ERR_INVALID_ARG, "no such session");
    if (p->lru) return lru_append(p, sid, k, v, n, st);
    if (s->state != KV_SESSION_ACTIVE) return fail(KV_ERR_BAD_STATE, "append to a paused session");
    if (n < 1) return fail(KV_ERR_INVALID_ARG, "n must be >= 1");
    if (!p->host_only && (!k || !v)) return fail(KV_ERR_INVALID_ARG, "null k or v");
    if ((reinterpret_cast<uintptr_t>(k) | reinterpret_cast<uintptr_t>(v)) & 15)
        return fail(KV_ERR_INVALID_ARG, "k and v must be 16-byte aligned");
    if (s->T + n > s->cap) return fail(KV_ERR_INVALID_ARG, "append past the session capacity");
    const int bt = p->cfg.block_tokens;
    const int64_t have = static_cast<int64_t>(s->blocks.size());
    const int64_t need = (s->T + n + bt - 1) / bt - have;
    if (need > static_cast<int64_t>(p->free_list.size()))
        return fail(KV_ERR_NO_HOT_BLOCKS, "hot pool has too few free blocks for the append");

    DeviceGuard dg(p->cfg.device, !p->host_only);
    std::vector<int32_t> fresh(need);
    for (int64_t i = 0; i < need; ++i) fresh[i] = p->free_list[p->free_list.size() - 1 - i];

    int rc = ensure_event(p, &s->appended);
    if (!rc && s->ready_recorded)
        rc = p->cuda("cudaStreamWaitEvent", [&] { return cudaStreamWaitEvent(st, s->ready, 0); });
    if (!rc && need > 0) rc = p->wait_fences(fresh.data(), fresh.size(), st);
    if (!rc && need > 0) rc = p->write_table(sid, fresh.data(), have, need, st);
    if (!rc) {
        kvt::AppendArgs a;
        a.k = static_cast<const uint8_t *>(k);
        a.v = static_cast<const uint8_t *>(v);
        a.table = p->d_tables + static_cast<int64_t>(sid) * p->table_stride;
        a.hot = static_cast<uint8_t *>(p->cfg.hot_base);
        a.pos0 = s->T;
        a.n = n;
        a.err = p->d_err;
        a.s = p->shape;
        rc = p->cuda("append launch", [&] { return kvt::launch_append(a, p->num_sms, st); });
    }
    if (!rc)
        rc = p->cuda("cudaEventRecord", [&] { return cudaEventRecord(s->appended, st); });
    if (rc) return rc;   // host state untouched

    p->free_list.resize(p->free_list.size() - need);
    p->clear_fences(fresh.data(), fresh.size());
    s->blocks.insert(s->blocks.end(), fresh.begin(), fresh.end());
    s->T += n;
    s->appended_recorded = !p->host_only;
    p->stats.free_blocks -= need;
    p->stats.used_blocks += need;
    p->stats.bytes_appended += static_cast<int64_t>(n) * p->token_bytes;
    p->stats.appends += 1;
    return KV_OK;
}

int decode_attention(kv_pool *p, int32_t layer, const void *q, const int32_t *block_tables,
                     const int32_t *seq_lens, int32_t B, int32_t max_blocks, float scale,
                     float *out, kv_stream_t stream_) {
    return decode_attention_ex(p, layer, q, block_tables, seq_lens, B, max_blocks, scale, out, 0u,
                               stream_);
}

static int decode_impl(kv_pool *p, int32_t layer, const void *q, const void *k_new,
                       const void *v_new, const int32_t *block_tables, const int32_t *seq_lens,
                       int32_t B, int32_t max_blocks, float scale, float *out, uint32_t flags,
                       kv_stream_t stream_) {
    if (flags & ~static_cast<uint32_t>(KV_DECODE_OVERLAP_PREVIOUS | KV_DECODE_OUT_BF16))
        return fail(KV_ERR_INVALID_ARG, "unknown decode flag");
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    if (!q || !block_tables || !seq_lens || !out) return fail(KV_ERR_INVALID_ARG, "null pointer");
    if (!decode_pointers_aligned(q, block_tables, seq_lens, out))
        return fail(KV_ERR_INVALID_ARG, "q, block_tables, seq_lens need 4-byte and out 16-byte alignment");
    if (layer < -1 || layer >= p->cfg.num_layers) return fail(KV_ERR_INVALID_ARG, "bad layer");
    const int nl = layer < 0 ? p->cfg.num_layers : 1;
    if (B < 1 || static_cast<int64_t>(nl) * B > 65535)
        return fail(KV_ERR_INVALID_ARG, "B out of range");
    if (max_blocks < 1 || max_blocks > (1 << 26))
        return fail(KV_ERR_INVALID_ARG, "max_blocks out of range");
    const int splits = kvt::max_splits_for(static_cast<int64_t>(max_blocks) * p->cfg.block_tokens);
    const int64_t rows = static_cast<int64_t>(nl) * B * p->cfg.num_q_heads * splits;
    if (rows > p->part_rows)
        return fail(KV_ERR_INVALID_ARG,
                    "decode workspace too small: layers x B x Hq x splits(max_blocks) exceeds "
                    "max_batch x Hq x splits(max_context)");
    if (!(scale == scale) || std::isinf(scale)) return fail(KV_ERR_INVALID_ARG, "scale not finite");
    // arguments first, then the pool's state
    if (p->host_only) return fail(KV_ERR_BAD_STATE, "decode_attention on a host-logic-only pool");
    DeviceGuard dg(p->cfg.device, true);
    kvt::DecodeArgs a;
    a.q = static_cast<const uint16_t *>(q);
    a.tables = block_tables;
    a.seq_lens = seq_lens;
    a.out = out;
    a.part_o = p->d_part_o;
    a.part_ml = p->d_part_ml;
    a.counters = p->d_counters;
    a.err = p->d_err;
    a.B = B;
    a.max_blocks = max_blocks;
    a.layer0 = layer < 0 ? 0 : layer;
    a.nlayers = nl;
    a.max_splits = splits;
    a.scale_log2 = scale * 1.4426950408889634f;
    a.out_bf16 = (flags & KV_DECODE_OUT_BF16) ? 1 : 0;
    a.k_new = static_cast<const uint16_t *>(k_new);
    a.v_new = static_cast<const uint16_t *>(v_new);
    a.hot = static_cast<uint16_t *>(p->cfg.hot_base);
    a.inject_extra_tx = p->inject_timeout ? 16 : 0;
    a.s = p->shape;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream_);
    const bool overlap = (flags & KV_DECODE_OVERLAP_PREVIOUS) != 0;
    int rc = p->cuda("decode launch", [&] { return kvt::launch_decode(p->tmap, a, p->num_sms, st, overlap); });
    if (rc) return rc;
    p->inject_timeout = false;
    p->stats.decodes += 1;
    return KV_OK;
}

int decode_attention_ex(kv_pool *p, int32_t layer, const void *q, const int32_t *block_tables,
                        const int32_t *seq_lens, int32_t B, int32_t max_blocks, float scale,
                        float *out, uint32_t flags, kv_stream_t stream) {
    return decode_impl(p, layer, q, nullptr, nullptr, block_tables, seq_lens, B, max_blocks,
                       scale, out, flags, stream);
}

int decode_append_attention(kv_pool *p, int32_t layer, const void *q, const void *k_new,
                            const void *v_new, const int32_t *block_tables,
                            const int32_t *seq_lens, int32_t B, int32_t max_blocks, float scale,
                            float *out, uint32_t flags, kv_stream_t stream) {
    if (!k_new || !v_new) return fail(KV_ERR_INVALID_ARG, "null k_new or v_new");
    if ((reinterpret_cast<uintptr_t>(k_new) | reinterpret_cast<uintptr_t>(v_new)) & 15)
        return fail(KV_ERR_INVALID_ARG, "k_new and v_new must be 16-byte aligned");
    return decode_impl(p, layer, q, k_new, v_new, block_tables, seq_lens, B, max_blocks, scale,
                       out, flags, stream);
}

int session_pause(kv_pool *p, int32_t sid, kv_stream_t stream_) {
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    Session *s = p->session(sid);
    if (!s) return fail(KV_ERR_INVALID_ARG, "no such session");
    if (s->state != KV_SESSION_ACTIVE) return fail(KV_ERR_BAD_STATE, "pause of a session that is not active");
    if (p->lru) {   // write-on-evict: nothing moves now; the blocks age in LRU order
        s->state = KV_SESSION_PAUSED;
        p->stats.pauses += 1;
        return KV_OK;
    }
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream_);
    DeviceGuard dg(p->cfg.device, !p->host_only);

    // Fence slot that will mark the freed blocks; its previous pack must be
    // complete before the slot is re-recorded.
    const int f = p->next_fence;
    int rc = KV_OK;
    if (p->fences[f].gen != 0)
        rc = p->cuda("cudaEventSynchronize", [&] { return cudaEventSynchronize(p->fences[f].ev); });
    if (!rc && s->appended_recorded)
        rc = p->cuda("cudaStreamWaitEvent", [&] { return cudaStreamWaitEvent(st, s->appended, 0); });
    if (!rc && s->ready_recorded)
        rc = p->cuda("cudaStreamWaitEvent", [&] { return cudaStreamWaitEvent(st, s->ready, 0); });
    const int64_t t0 = s->cold_valid, t1 = s->T;
    if (!rc && t1 > t0) {
        kvt::MigArgs m = p->mig_args(sid, *s);
        m.t_begin = static_cast<int32_t>(t0);
        m.t_end = static_cast<int32_t>(t1);
        rc = p->cuda("pack launch", [&] { return kvt::launch_pack(m, p->num_sms, p->mig_ctas, st); });
    }
    if (!rc) rc = p->cuda("cudaEventRecord", [&] { return cudaEventRecord(p->fences[f].ev, st); });
    if (rc) return rc;

    p->next_fence = (f + 1) % kFenceSlots;
    const uint64_t gen = ++p->fence_gen;
    p->fences[f].gen = gen;
    s->pack_fence = static_cast<int16_t>(f);
    s->pack_gen = gen;
    for (int32_t b : s->blocks) {
        p->free_list.push_back(b);
        p->block_fence[b] = static_cast<int16_t>(f);
        p->block_fence_gen[b] = gen;
    }
    p->stats.free_blocks += static_cast<int64_t>(s->blocks.size());
    p->stats.used_blocks -= static_cast<int64_t>(s->blocks.size());
    p->stats.bytes_packed += (t1 - t0) * p->token_bytes;
    p->stats.pauses += 1;
    s->blocks.clear();
    s->cold_valid = t1;
    s->state = KV_SESSION_PAUSED;
    s->ready_recorded = false;
    s->appended_recorded = false;
    return KV_OK;
}

int session_resume(kv_pool *p, int32_t sid, kv_stream_t stream_) {
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    Session *s = p->session(sid);
    if (!s) return fail(KV_ERR_INVALID_ARG, "no such session");
    if (s->state != KV_SESSION_PAUSED) return fail(KV_ERR_BAD_STATE, "resume of a session that is not paused");
    if (p->lru) return lru_resume(p, sid, reinterpret_cast<cudaStream_t>(stream_));
    const int bt = p->cfg.block_tokens;
    const int64_t need = (s->T + bt - 1) / bt;
    if (need > static_cast<int64_t>(p->free_list.size()))
        return fail(KV_ERR_NO_HOT_BLOCKS, "hot pool has too few free blocks for the resume");
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream_);
    DeviceGuard dg(p->cfg.device, !p->host_only);
    std::vector<int32_t> fresh(need);
    for (int64_t i = 0; i < need; ++i) fresh[i] = p->free_list[p->free_list.size() - 1 - i];

    int rc = ensure_event(p, &s->ready);
    if (!rc) rc = p->wait_fences(fresh.data(), fresh.size(), st);
    // The session's own last pack reads the table row this resume rewrites:
    // order after it while its fence slot still holds that pack (a re-recorded
    // slot means it was synchronised first).
    if (!rc && s->pack_fence >= 0 && p->fences[s->pack_fence].gen == s->pack_gen)
        rc = p->cuda("cudaStreamWaitEvent",
                     [&] { return cudaStreamWaitEvent(st, p->fences[s->pack_fence].ev, 0); });
    if (!rc && need == 0) {
        // an empty session: no blocks, nothing to copy
    } else if (!rc && need <= kvt::kResumeInlineMax) {
        // one launch: the block ids ride in the parameters, the kernel writes the row
        kvt::ResumeArgs r;
        r.m = p->mig_args(sid, *s);
        r.m.t_begin = 0;
        r.m.t_end = static_cast<int32_t>(s->T);
        r.n = static_cast<int32_t>(need);
        r.pad = 0;
        std::memcpy(r.blocks, fresh.data(), sizeof(int32_t) * need);
        rc = p->cuda("unpack launch",
                     [&] { return kvt::launch_unpack_inline(r, p->num_sms, p->mig_ctas, st); });
    } else if (!rc) {
        rc = p->write_table(sid, fresh.data(), 0, need, st);
        if (!rc) {
            kvt::MigArgs m = p->mig_args(sid, *s);
            m.t_begin = 0;
            m.t_end = static_cast<int32_t>(s->T);
            rc = p->cuda("unpack launch",
                         [&] { return kvt::launch_unpack(m, p->num_sms, p->mig_ctas, st); });
        }
    }
    if (!rc) rc = p->cuda("cudaEventRecord", [&] { return cudaEventRecord(s->ready, st); });
    if (rc) return rc;

    p->free_list.resize(p->free_list.size() - need);
    p->clear_fences(fresh.data(), fresh.size());
    s->blocks = fresh;
    s->state = KV_SESSION_ACTIVE;
    s->ready_recorded = !p->host_only;
    p->stats.free_blocks -= need;
    p->stats.used_blocks += need;
    p->stats.bytes_unpacked += s->T * p->token_bytes;
    p->stats.resumes += 1;
    return KV_OK;
}

int session_ready_event(kv_pool *p, int32_t sid, kv_event_t *ev) {
    if (!p || !ev) return fail(KV_ERR_INVALID_ARG, "null argument");
    Session *s = p->session(sid);
    if (!s) return fail(KV_ERR_INVALID_ARG, "no such session");
    *ev = s->ready_recorded ? reinterpret_cast<kv_event_t>(s->ready) : nullptr;
    return KV_OK;
}

int session_info(kv_pool *p, int32_t sid, kv_session_info *out) {
    if (!p || !out) return fail(KV_ERR_INVALID_ARG, "null argument");
    Session *s = p->session(sid);
    if (!s) return fail(KV_ERR_INVALID_ARG, "no such session");
    out->state = s->state;
    out->num_blocks = static_cast<int32_t>(p->lru ? s->hot_count : static_cast<int64_t>(s->blocks.size()));
    out->tokens = s->T;
    out->capacity = s->cap;
    out->cold_valid = s->cold_valid;
    out->image = p->host_only ? nullptr : static_cast<uint8_t *>(p->cfg.cold_base) + s->img_off;
    return KV_OK;
}

int session_block_table(kv_pool *p, int32_t sid, int32_t *host_row, int32_t cap, int32_t *nblocks) {
    if (!p || !nblocks || (cap > 0 && !host_row)) return fail(KV_ERR_INVALID_ARG, "null argument");
    Session *s = p->session(sid);
    if (!s) return fail(KV_ERR_INVALID_ARG, "no such session");
    *nblocks = static_cast<int32_t>(s->blocks.size());
    const int32_t n = std::min<int32_t>(cap, *nblocks);
    if (n > 0) std::memcpy(host_row, s->blocks.data(), sizeof(int32_t) * n);
    return KV_OK;
}

int session_block_table_device(kv_pool *p, int32_t sid, const int32_t **dev_row,
                               int32_t *nblocks) {
    if (!p || !dev_row || !nblocks) return fail(KV_ERR_INVALID_ARG, "null argument");
    Session *s = p->session(sid);
    if (!s) return fail(KV_ERR_INVALID_ARG, "no such session");
    if (p->host_only) return fail(KV_ERR_BAD_STATE, "host-logic-only pools have no device tables");
    *dev_row = p->d_tables + static_cast<int64_t>(sid) * p->table_stride;
    *nblocks = static_cast<int32_t>(s->blocks.size());
    return KV_OK;
}

// Device inputs of a decode batch from the pool's tables: row b of
// block_tables (entries past the session's length set to -1) and seq_lens.
// lens / nblk / new_blk, when given, replace the sessions' current lengths
// and row sizes (a call that launches before committing its host state).
static int gather_batch(kv_pool *p, const int32_t *sids, int32_t B, int32_t *block_tables,
                        int32_t max_blocks, int32_t *seq_lens, cudaStream_t st,
                        const int32_t *lens = nullptr, const int32_t *nblk = nullptr,
                        const int32_t *new_blk = nullptr) {
    for (int32_t r0 = 0; r0 < B; r0 += kvt::kGatherMax) {
        kvt::GatherArgs a;
        a.arena = p->d_tables;
        a.stride = p->table_stride;
        a.tables = block_tables;
        a.seq_lens = seq_lens;
        a.max_blocks = max_blocks;
        a.row0 = r0;
        a.count = std::min(B - r0, kvt::kGatherMax);
        for (int32_t i = 0; i < a.count; ++i) {
            const Session &s = p->sessions[sids[r0 + i]];
            a.sids[i] = sids[r0 + i];
            a.lens[i] = lens ? lens[r0 + i] : static_cast<int32_t>(s.T);
            a.nblk[i] = nblk ? nblk[r0 + i] : static_cast<int32_t>(s.blocks.size());
            a.new_blk[i] = new_blk ? new_blk[r0 + i] : -1;
        }
        int rc = p->cuda("gather launch", [&] { return kvt::launch_gather(a, st); });
        if (rc) return rc;
    }
    return KV_OK;
}

int kv_pool_batch_tables(kv_pool *p, const int32_t *sids, int32_t B, int32_t *block_tables,
                         int32_t max_blocks, int32_t *seq_lens, kv_stream_t stream_) {
    if (!p || !sids || B < 1) return fail(KV_ERR_INVALID_ARG, "bad argument");
    if (p->host_only && !p->lru)
        return fail(KV_ERR_BAD_STATE, "batch tables on a host-logic-only pool");
    if (!p->host_only && (!block_tables || !seq_lens)) return fail(KV_ERR_INVALID_ARG, "null output");
    if ((reinterpret_cast<uintptr_t>(block_tables) | reinterpret_cast<uintptr_t>(seq_lens)) & 3)
        return fail(KV_ERR_INVALID_ARG, "block_tables and seq_lens must be 4-byte aligned");
    if (max_blocks < 1) return fail(KV_ERR_INVALID_ARG, "max_blocks must be >= 1");
    for (int32_t i = 0; i < B; ++i) {
        Session *s = p->session(sids[i]);
        if (!s) return fail(KV_ERR_INVALID_ARG, "no such session in batch");
        if (s->state != KV_SESSION_ACTIVE) return fail(KV_ERR_BAD_STATE, "paused session in batch");
        if (s->T < 1) return fail(KV_ERR_INVALID_ARG, "empty session in batch");
        if (static_cast<int64_t>(s->blocks.size()) > max_blocks)
            return fail(KV_ERR_INVALID_ARG, "max_blocks shorter than a session's table");
    }
    DeviceGuard dg(p->cfg.device, true);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream_);
    if (p->lru) {
        int rc = lru_fetch_batch(p, sids, B, st);
        if (rc || p->host_only) return rc;   // host-logic pools: bookkeeping only
    }
    return gather_batch(p, sids, B, block_tables, max_blocks, seq_lens, st);
}

// Path 3 for one decode step: every member gets position T (a fresh block
// when its tail block is full) and, in residency mode, its evicted blocks
// back; victims come only from sessions outside the batch. The values
// arrive with decode_append_attention. Free-list pops go in batch order:
// a member's missing blocks (ascending), then its fresh block.
int kv_pool_batch_reserve(kv_pool *p, const int32_t *sids, int32_t B, int32_t *block_tables,
                          int32_t max_blocks, int32_t *seq_lens, kv_stream_t stream_) {
    if (!p || !sids || B < 1) return fail(KV_ERR_INVALID_ARG, "bad argument");
    if (!p->host_only && (!block_tables || !seq_lens)) return fail(KV_ERR_INVALID_ARG, "null output");
    if ((reinterpret_cast<uintptr_t>(block_tables) | reinterpret_cast<uintptr_t>(seq_lens)) & 3)
        return fail(KV_ERR_INVALID_ARG, "block_tables and seq_lens must be 4-byte aligned");
    if (max_blocks < 1) return fail(KV_ERR_INVALID_ARG, "max_blocks must be >= 1");
    const int bt = p->cfg.block_tokens;
    const std::vector<int32_t> members(sids, sids + B);
    for (int32_t i = 0; i < B; ++i) {
        Session *s = p->session(sids[i]);
        if (!s) return fail(KV_ERR_INVALID_ARG, "no such session in batch");
        if (std::find(members.begin(), members.begin() + i, sids[i]) != members.begin() + i)
            return fail(KV_ERR_INVALID_ARG, "a session appears twice in the batch");
        if (s->state != KV_SESSION_ACTIVE) return fail(KV_ERR_BAD_STATE, "paused session in batch");
        if (s->T + 1 > s->cap) return fail(KV_ERR_INVALID_ARG, "append past the session capacity");
        if ((s->T + bt) / bt > max_blocks)
            return fail(KV_ERR_INVALID_ARG, "max_blocks shorter than a session's table");
    }
    std::vector<std::vector<int32_t>> miss(B);
    std::vector<char> grow(B);
    int64_t need = 0;
    for (int32_t i = 0; i < B; ++i) {
        const Session &s = p->sessions[sids[i]];
        if (p->lru)
            for (size_t j = 0; j < s.blocks.size(); ++j)
                if (s.blocks[j] < 0) miss[i].push_back(static_cast<int32_t>(j));
        grow[i] = (s.T % bt) == 0;
        need += static_cast<int64_t>(miss[i].size()) + grow[i];
    }
    std::vector<Victim> vic;
    if (p->lru ? !p->plan_evict(need, members, vic)
               : need > static_cast<int64_t>(p->free_list.size()))
        return fail(KV_ERR_NO_HOT_BLOCKS, "the batch's blocks and new positions do not fit in the hot pool");
    const std::vector<int32_t> got = p->peek_alloc(need, vic);
    std::vector<std::vector<int32_t>> rows(B);
    std::vector<kvt::BlockJob> jobs;
    std::vector<int32_t> fresh;      // popped slots that are not eviction victims
    int64_t k = 0, fetched = 0;
    for (int32_t i = 0; i < B; ++i) {
        const Session &s = p->sessions[sids[i]];
        rows[i] = s.blocks;
        for (int32_t j : miss[i]) {
            rows[i][j] = got[k];
            jobs.push_back(p->fetch_job(sids[i], j, got[k], 0, p->tokens_in_block(s, j)));
            fetched += p->tokens_in_block(s, j);
            ++k;
        }
        if (grow[i]) rows[i].push_back(got[k++]);
    }
    // Slots that come off the free list (not from this call's victims) may
    // have been freed by a pause whose pack is still running.
    for (int64_t i = 0; i < need && i < static_cast<int64_t>(p->free_list.size()); ++i)
        fresh.push_back(p->free_list[p->free_list.size() - 1 - i]);

    DeviceGuard dg(p->cfg.device, !p->host_only);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream_);
    int rc = KV_OK;
    for (int32_t i = 0; !rc && i < B; ++i) {
        const Session &s = p->sessions[sids[i]];
        if (s.ready_recorded) rc = wait_event(p, st, s.ready);
    }
    if (!rc && !fresh.empty()) rc = p->wait_fences(fresh.data(), fresh.size(), st);
    if (!rc) rc = p->evict_device(vic, st);
    for (int32_t i = 0; !rc && i < B; ++i)
        if (!miss[i].empty()) rc = p->wait_packed(sids[i], st);
    if (!rc) rc = p->run_jobs(jobs, false, st);
    // Fetched entries were written by their jobs; a new tail block's entry is
    // written by the gather launch below (host-logic pools launch nothing).
    std::vector<int32_t> new_blk(B, -1), lens(B), nblk(B);
    for (int32_t i = 0; i < B; ++i) {
        if (grow[i]) new_blk[i] = rows[i].back();
        lens[i] = static_cast<int32_t>(p->sessions[sids[i]].T + 1);
        nblk[i] = static_cast<int32_t>(rows[i].size());
    }
    if (!rc && !p->host_only)
        rc = gather_batch(p, sids, B, block_tables, max_blocks, seq_lens, st, lens.data(),
                          nblk.data(), new_blk.data());
    if (rc) return rc;   // host state untouched

    p->evict_commit(vic);
    p->free_list.resize(p->free_list.size() - need);
    p->clear_fences(fresh.data(), fresh.size());
    const uint64_t stamp = ++p->clock;
    for (int32_t i = 0; i < B; ++i) {
        Session &s = p->sessions[sids[i]];
        if (p->lru) p->lru_out(sids[i]);
        s.blocks = rows[i];
        if (grow[i] && p->lru) s.img_tok.push_back(0);
        s.T += 1;
        if (p->lru) {
            s.hot_count += static_cast<int64_t>(miss[i].size()) + grow[i];
            s.last_use = stamp;
            p->lru_in(sids[i]);
        }
    }
    p->stats.free_blocks -= need;
    p->stats.used_blocks += need;
    p->stats.bytes_unpacked += fetched * p->token_bytes;
    p->stats.batch_blocks_fetched += static_cast<int64_t>(jobs.size());
    p->stats.bytes_appended += static_cast<int64_t>(B) * p->token_bytes;
    p->stats.appends += B;
    return KV_OK;
}

// One step ahead of decode (Section 3, "Eviction, resume and decode": decode
// reads a known set of blocks, so the next step's can be fetched while the
// current step runs). Victims come from sessions in neither the next batch
// nor `busy`, the batch the current step is still reading.
int kv_pool_prefetch(kv_pool *p, const int32_t *sids, int32_t B, const int32_t *busy,
                     int32_t n_busy, kv_stream_t stream_) {
    if (!p || !sids || B < 1 || n_busy < 0 || (n_busy > 0 && !busy))
        return fail(KV_ERR_INVALID_ARG, "bad argument");
    for (int32_t i = 0; i < B; ++i) {
        Session *s = p->session(sids[i]);
        if (!s) return fail(KV_ERR_INVALID_ARG, "no such session in the next batch");
        if (s->state != KV_SESSION_ACTIVE)
            return fail(KV_ERR_BAD_STATE, "paused session in the next batch");
    }
    for (int32_t i = 0; i < n_busy; ++i)
        if (!p->session(busy[i])) return fail(KV_ERR_INVALID_ARG, "no such session in busy");
    if (!p->lru) return KV_OK;   // simple mode: an active session's blocks are always hot
    const std::vector<int32_t> uniq = unique_ids(sids, B);
    std::vector<int32_t> protect(uniq);
    for (int32_t i = 0; i < n_busy; ++i)
        if (std::find(protect.begin(), protect.end(), busy[i]) == protect.end())
            protect.push_back(busy[i]);
    DeviceGuard dg(p->cfg.device, !p->host_only);
    int64_t blocks = 0;
    int rc = lru_fetch(p, uniq, protect, true, reinterpret_cast<cudaStream_t>(stream_), &blocks);
    if (rc) return rc;
    p->stats.blocks_prefetched += blocks;
    p->stats.prefetches += 1;
    return KV_OK;
}

int kv_pool_shuffle_free(kv_pool *p, uint64_t seed) {
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    fisher_yates(p->free_list, p->free_list.size(), seed);
    return KV_OK;
}

int kv_pool_free_list(kv_pool *p, int32_t *host_out, int64_t cap, int64_t *n) {
    if (!p || !n || (cap > 0 && !host_out)) return fail(KV_ERR_INVALID_ARG, "null argument");
    *n = static_cast<int64_t>(p->free_list.size());
    const int64_t m = std::min<int64_t>(cap, *n);
    if (m > 0) std::memcpy(host_out, p->free_list.data(), sizeof(int32_t) * m);
    return KV_OK;
}

int kv_pool_get_stats(kv_pool *p, kv_pool_stats *out) {
    if (!p || !out) return fail(KV_ERR_INVALID_ARG, "null argument");
    *out = p->stats;
    out->cold_bytes_used = p->cold_used;
    return KV_OK;
}

int kv_pool_check_device(kv_pool *p, int32_t *flags) {
    if (!p || !flags) return fail(KV_ERR_INVALID_ARG, "null argument");
    *flags = 0;
    if (p->host_only) return KV_OK;
    DeviceGuard dg(p->cfg.device, true);
    int rc = p->cuda("cudaDeviceSynchronize", [&] { return cudaDeviceSynchronize(); });
    if (!rc) rc = p->cuda("cudaMemcpy", [&] {
        return cudaMemcpy(flags, p->d_err, 4, cudaMemcpyDeviceToHost);
    });
    if (!rc) rc = p->cuda("cudaMemset", [&] { return cudaMemset(p->d_err, 0, 4); });
    // Every decode call leaves the split-arrival counters at zero; any other
    // value comes from calls that overlapped on the GPU.
    std::vector<int32_t> cnt(static_cast<size_t>(p->counter_count));
    if (!rc && !cnt.empty())
        rc = p->cuda("cudaMemcpy", [&] {
            return cudaMemcpy(cnt.data(), p->d_counters, cnt.size() * 4, cudaMemcpyDeviceToHost);
        });
    if (rc) return rc;
    bool stale = false;
    for (int32_t v : cnt) stale |= v != 0;
    if (stale) {
        rc = p->cuda("cudaMemset", [&] { return cudaMemset(p->d_counters, 0, cnt.size() * 4); });
        if (rc) return rc;
        *flags |= KV_DEVICE_STALE_COUNTERS;
    }
    if (*flags) return fail(KV_ERR_DEVICE_CHECK, "a device check fired (flags " + std::to_string(*flags) + ")");
    return KV_OK;
}

int kv_pool_set_migration_limit(kv_pool *p, int32_t max_ctas) {
    if (!p || max_ctas < 0) return fail(KV_ERR_INVALID_ARG, "bad argument");
    p->mig_ctas = max_ctas;
    return KV_OK;
}

int kv_pool_inject_cuda_failure(kv_pool *p, int32_t n) {
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    p->inject_countdown = n > 0 ? n : 0;
    return KV_OK;
}

int kv_pool_inject_decode_timeout(kv_pool *p, int32_t on) {
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    p->inject_timeout = on != 0;
    return KV_OK;
}

int kv_pool_inject_stale_counter(kv_pool *p) {
    if (!p) return fail(KV_ERR_INVALID_ARG, "null pool");
    if (p->host_only) return fail(KV_ERR_BAD_STATE, "no device workspace on a host-logic pool");
    DeviceGuard dg(p->cfg.device, true);
    const int32_t one = 1;
    int rc = p->cuda("cudaDeviceSynchronize", [&] { return cudaDeviceSynchronize(); });
    if (!rc) rc = p->cuda("cudaMemcpy", [&] {
        return cudaMemcpy(p->d_counters, &one, 4, cudaMemcpyHostToDevice);
    });
    return rc;
}

}  // extern "C"
