/* A plain C caller of libkvtier.so, compiled and run by tests/test_c_consumer.py.
 *
 * It uses only include/kvtier.h: a host-logic-only pool (no GPU, no arenas)
 * with the paper's KV shape, two sessions, appends across a block boundary,
 * one batch reservation, a pause and a resume, and a few calls that must fail.
 * It prints key=value lines; the test compares the block ids with the oracle's
 * free-list contract. Written to compile as C99 and as C++.
 */
#include <stdio.h>
#include <string.h>

#include "kvtier.h"

static int failures = 0;

static void expect_code(const char *what, int got, int want) {
    if (got != want) {
        printf("mismatch %s: got %d want %d (%s)\n", what, got, want, kv_last_error());
        ++failures;
    }
}

static void print_row(kv_pool *pool, int32_t sid, const char *key) {
    int32_t row[64];
    int32_t n = 0;
    int32_t i;
    expect_code("session_block_table", session_block_table(pool, sid, row, 64, &n), KV_OK);
    printf("%s=", key);
    for (i = 0; i < n; ++i) printf(i ? ",%d" : "%d", (int)row[i]);
    printf("\n");
}

int main(void) {
    kv_pool_config cfg;
    kv_pool_config bad;
    kv_pool *pool = NULL;
    kv_pool *none = NULL;
    kv_session_info info;
    kv_pool_stats st;
    int32_t s0 = -1, s1 = -1;
    int32_t batch[2];
    float scratch[8];
    /* a 16-byte-aligned stand-in for the device buffers (never dereferenced on
       a host-logic pool) */
    float *out_dummy = (float *)(((uintptr_t)scratch + 15) & ~(uintptr_t)15);

    memset(&cfg, 0, sizeof cfg);
    cfg.num_layers = 48;
    cfg.num_q_heads = 32;
    cfg.num_kv_heads = 4;
    cfg.head_dim = 128;
    cfg.block_tokens = 16;
    cfg.max_sessions = 4;
    cfg.max_batch = 4;
    cfg.device = 0;
    cfg.max_context = 1024;
    cfg.num_hot_blocks = 20;
    cfg.cold_bytes = (int64_t)4 * 1024 * 98304;
    cfg.alloc_seed = 7;
    cfg.flags = KV_POOL_HOST_LOGIC_ONLY;

    printf("token_bytes=%lld\n", (long long)kv_token_bytes(&cfg));
    printf("block_bytes=%lld\n", (long long)kv_block_bytes(&cfg));

    expect_code("kv_pool_create", kv_pool_create(&cfg, &pool), KV_OK);
    if (!pool) {
        printf("failures=%d\n", failures + 1);
        return 1;
    }
    expect_code("session_create 0", session_create(pool, 200, &s0), KV_OK);
    expect_code("session_create 1", session_create(pool, 200, &s1), KV_OK);
    printf("sids=%d,%d\n", (int)s0, (int)s1);

    expect_code("append 40", session_append(pool, s0, NULL, NULL, 40, NULL), KV_OK);
    expect_code("append 16", session_append(pool, s1, NULL, NULL, 16, NULL), KV_OK);
    print_row(pool, s0, "row0_after_append");
    print_row(pool, s1, "row1_after_append");

    batch[0] = s0;
    batch[1] = s1;
    expect_code("batch_reserve", kv_pool_batch_reserve(pool, batch, 2, NULL, 64, NULL, NULL), KV_OK);
    print_row(pool, s1, "row1_after_reserve");
    expect_code("session_info", session_info(pool, s0, &info), KV_OK);
    printf("tokens0=%lld\n", (long long)info.tokens);

    expect_code("pause", session_pause(pool, s0, NULL), KV_OK);
    expect_code("resume", session_resume(pool, s0, NULL), KV_OK);
    print_row(pool, s0, "row0_after_resume");

    /* calls that must fail and leave a message */
    expect_code("resume active", session_resume(pool, s0, NULL), KV_ERR_BAD_STATE);
    printf("last_error_nonempty=%d\n", kv_last_error()[0] != '\0');
    expect_code("decode on host-logic pool",
                decode_attention(pool, 0, out_dummy, batch, batch, 1, 1, 1.0f, out_dummy, NULL),
                KV_ERR_BAD_STATE);
    expect_code("decode with misaligned out",
                decode_attention(pool, 0, out_dummy, batch, batch, 1, 1, 1.0f, out_dummy + 1, NULL),
                KV_ERR_INVALID_ARG);
    expect_code("append past capacity", session_append(pool, s1, NULL, NULL, 500, NULL),
                KV_ERR_INVALID_ARG);
    {
        const int32_t *dev_row = NULL;
        int32_t nb = 0;
        expect_code("device table row on a host-logic pool",
                    session_block_table_device(pool, s0, &dev_row, &nb), KV_ERR_BAD_STATE);
    }
    {
        int32_t flags = -1;
        expect_code("device check on a host-logic pool", kv_pool_check_device(pool, &flags), KV_OK);
        if (flags != 0) {
            fprintf(stderr, "device check on a host-logic pool: flags %d\n", flags);
            ++failures;
        }
        expect_code("stale-counter hook on a host-logic pool", kv_pool_inject_stale_counter(pool),
                    KV_ERR_BAD_STATE);
    }
    batch[1] = s0;
    expect_code("session twice in a batch",
                kv_pool_batch_reserve(pool, batch, 2, NULL, 64, NULL, NULL), KV_ERR_INVALID_ARG);
    bad = cfg;
    bad.head_dim = 64;
    expect_code("head_dim 64", kv_pool_create(&bad, &none), KV_ERR_INVALID_ARG);

    expect_code("stats", kv_pool_get_stats(pool, &st), KV_OK);
    printf("free_blocks=%lld used_blocks=%lld appends=%lld pauses=%lld resumes=%lld\n",
           (long long)st.free_blocks, (long long)st.used_blocks, (long long)st.appends,
           (long long)st.pauses, (long long)st.resumes);
    expect_code("destroy", kv_pool_destroy(pool), KV_OK);
    printf("failures=%d\n", failures);
    return failures ? 1 : 0;
}
