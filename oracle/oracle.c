/*
 * CPU oracle for the hot/cold KV tiering hot path.
 *
 * TEST INFRASTRUCTURE ONLY. Tests, the package's smoke check and the
 * benchmark's CPU-baseline leg call it; the CUDA library never does. It
 * shares no source, header, table or helper with that library.
 *
 * What it computes, and where the paper defines it
 * (Baek et al., "Hot-Cold Tiering of HBM and High Bandwidth Flash for Agentic
 * LLM Serving"):
 *
 *  - oracle_paged_decode: one decode step of attention over the cached KV of
 *    each session (Section 2, "Large Language Models": decoding attends to
 *    past KV held in fixed-size blocks; Section 3 data path 1). Paging does
 *    not change the mathematics, so this is the textbook definition, taken in
 *    double precision: s_i = scale * <q_h, k_i> for the session's tokens
 *    i = 0 .. seq_len-1 in logical order, p = softmax(s) computed in two
 *    passes (max, then sum of exp), out_h = sum_i p_i v_i. Query head h reads
 *    kv head h / (Hq / Hkv) (grouped-query attention, contiguous groups). Key
 *    i is fetched through the block table: block table[i / bt], slot i % bt.
 *  - oracle_unpack / oracle_pack: the resume (data path 2) and eviction (data
 *    path 4) copies between a session's contiguous layer-major cold image
 *    img[L][2][Hkv][T_cap][D] and its hot blocks hot[NB][L][2][Hkv][bt][D].
 *    Pack moves only tokens [t0, T): KV is immutable, so tokens already in
 *    the image are never rewritten (Section 3, "Memory hierarchy and write
 *    policy": write-on-evict writes each block at most once).
 *  - oracle_append: fresh KV written into the hot blocks (data path 3).
 *  - oracle_splitmix64 / free-list functions: the seeded placement of hot
 *    blocks. The paper does not define placement; the library's contract is
 *    a free list shuffled by Fisher-Yates driven by splitmix64 (Steele, Lea,
 *    Flood, OOPSLA 2014), blocks popped from the end of the list, freed
 *    blocks pushed back in logical order.
 *
 * Pins (tests/test_oracle_pins.py): dense attention through numpy/scipy on
 * tiny inputs, the 1-token and equal-key closed forms, invariance under
 * permutation of physical blocks, Hq = Hkv, NaN-poisoned tails, pack/unpack
 * round trips against a numpy reshape of the image, published splitmix64
 * outputs, and the paper's size arithmetic (96 KiB per token, 1.5 MiB per
 * block).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static double bf16_value(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Offset of element (blk, l, kv, g, slot, d) of the hot pool. */
static int64_t hot_offset(int64_t blk, int l, int kv, int g, int slot, int d,
                          int L, int Hkv, int D, int bt)
{
    return ((((blk * L + l) * 2 + kv) * Hkv + g) * (int64_t)bt + slot) * D + d;
}

/* Offset of element (l, kv, g, t, d) of a cold image with capacity T_cap. */
static int64_t img_offset(int l, int kv, int g, int64_t t, int d,
                          int Hkv, int D, int64_t T_cap)
{
    return ((((int64_t)l * 2 + kv) * Hkv + g) * T_cap + t) * D + d;
}

int oracle_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Bytes of K plus V per token over all layers: L x {K,V} x Hkv x D x 2 B. */
int64_t oracle_kv_bytes_per_token(int L, int Hkv, int D)
{
    return (int64_t)L * 2 * Hkv * D * 2;
}

/*
 * q:      [nlayers][B][Hq][D] bf16 bits, layer index relative to layer0
 * tables: [B][max_blocks] physical block ids
 * out:    [nlayers][B][Hq][D] double
 * Returns 0, or -1 for a bad argument (seq_len < 1, a table entry outside the
 * pool, a sequence longer than its table row).
 */
int oracle_paged_decode(const uint16_t *hot, int64_t num_blocks, int L, int Hq, int Hkv,
                        int D, int bt, int layer0, int nlayers, const uint16_t *q,
                        const int32_t *tables, int max_blocks, const int32_t *seq_lens,
                        int B, double scale, double *out, int nthreads)
{
    if (Hkv <= 0 || Hq % Hkv != 0 || layer0 < 0 || layer0 + nlayers > L)
        return -1;
    for (int b = 0; b < B; ++b) {
        int T = seq_lens[b];
        if (T < 1 || (int64_t)(T + bt - 1) / bt > max_blocks)
            return -1;
        for (int j = 0; j < (T + bt - 1) / bt; ++j) {
            int32_t p = tables[(int64_t)b * max_blocks + j];
            if (p < 0 || p >= num_blocks)
                return -1;
        }
    }
    const int group = Hq / Hkv;
    const int64_t tasks = (int64_t)nlayers * B * Hq;
    if (nthreads <= 0)
        nthreads = oracle_threads();
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads)
    for (int64_t task = 0; task < tasks; ++task) {
        const int h = (int)(task % Hq);
        const int b = (int)((task / Hq) % B);
        const int li = (int)(task / ((int64_t)Hq * B));
        const int l = layer0 + li;
        const int g = h / group;
        const int T = seq_lens[b];
        const int32_t *row = tables + (int64_t)b * max_blocks;
        const uint16_t *qh = q + (((int64_t)li * B + b) * Hq + h) * D;
        double *o = out + (((int64_t)li * B + b) * Hq + h) * D;
        double *s = (double *)malloc(sizeof(double) * (size_t)T);
        double *qd = (double *)malloc(sizeof(double) * (size_t)D);
        for (int d = 0; d < D; ++d)
            qd[d] = bf16_value(qh[d]);
        /* scores, logical order */
        for (int i = 0; i < T; ++i) {
            const uint16_t *k = hot + hot_offset(row[i / bt], l, 0, g, i % bt, 0, L, Hkv, D, bt);
            double acc = 0.0;
            for (int d = 0; d < D; ++d)
                acc += qd[d] * bf16_value(k[d]);
            s[i] = scale * acc;
        }
        /* softmax: pass 1 max, pass 2 normaliser */
        double m = s[0];
        for (int i = 1; i < T; ++i)
            if (s[i] > m)
                m = s[i];
        double z = 0.0;
        for (int i = 0; i < T; ++i) {
            s[i] = exp(s[i] - m);
            z += s[i];
        }
        for (int d = 0; d < D; ++d)
            o[d] = 0.0;
        for (int i = 0; i < T; ++i) {
            const uint16_t *v = hot + hot_offset(row[i / bt], l, 1, g, i % bt, 0, L, Hkv, D, bt);
            const double p = s[i] / z;
            for (int d = 0; d < D; ++d)
                o[d] += p * bf16_value(v[d]);
        }
        free(qd);
        free(s);
    }
    return 0;
}

/*
 * Resume copy: tokens [0, T) of the image into the session's hot blocks
 * (table_row[j] holds tokens j*bt .. j*bt+bt-1). Slots past T are not written.
 */
int oracle_unpack(const uint16_t *img, int64_t T_cap, int64_t T, const int32_t *table_row,
                  uint16_t *hot, int64_t num_blocks, int L, int Hkv, int D, int bt)
{
    if (T < 0 || T > T_cap)
        return -1;
    for (int64_t t = 0; t < T; ++t) {
        int32_t p = table_row[t / bt];
        if (p < 0 || p >= num_blocks)
            return -1;
        for (int l = 0; l < L; ++l)
            for (int kv = 0; kv < 2; ++kv)
                for (int g = 0; g < Hkv; ++g)
                    for (int d = 0; d < D; ++d)
                        hot[hot_offset(p, l, kv, g, (int)(t % bt), d, L, Hkv, D, bt)] =
                            img[img_offset(l, kv, g, t, d, Hkv, D, T_cap)];
    }
    return 0;
}

/*
 * Eviction copy: tokens [t0, T) of the hot blocks into the image. Returns the
 * number of image bytes written (0 when t0 >= T), or -1 for a bad argument.
 */
int64_t oracle_pack(const uint16_t *hot, int64_t num_blocks, const int32_t *table_row,
                    int64_t t0, int64_t T, uint16_t *img, int64_t T_cap, int L, int Hkv,
                    int D, int bt)
{
    if (t0 < 0 || T > T_cap)
        return -1;
    int64_t written = 0;
    for (int64_t t = t0; t < T; ++t) {
        int32_t p = table_row[t / bt];
        if (p < 0 || p >= num_blocks)
            return -1;
        for (int l = 0; l < L; ++l)
            for (int kv = 0; kv < 2; ++kv)
                for (int g = 0; g < Hkv; ++g)
                    for (int d = 0; d < D; ++d) {
                        img[img_offset(l, kv, g, t, d, Hkv, D, T_cap)] =
                            hot[hot_offset(p, l, kv, g, (int)(t % bt), d, L, Hkv, D, bt)];
                        written += 2;
                    }
    }
    return written;
}

/*
 * Fresh-KV write: token n_i of k/v ([L][n][Hkv][D]) goes to logical position
 * pos0 + n_i of the session.
 */
int oracle_append(uint16_t *hot, int64_t num_blocks, const int32_t *table_row, int64_t pos0,
                  int n, const uint16_t *k, const uint16_t *v, int L, int Hkv, int D, int bt)
{
    for (int i = 0; i < n; ++i) {
        int64_t t = pos0 + i;
        int32_t p = table_row[t / bt];
        if (p < 0 || p >= num_blocks)
            return -1;
        for (int l = 0; l < L; ++l)
            for (int g = 0; g < Hkv; ++g)
                for (int d = 0; d < D; ++d) {
                    int64_t src = (((int64_t)l * n + i) * Hkv + g) * D + d;
                    hot[hot_offset(p, l, 0, g, (int)(t % bt), d, L, Hkv, D, bt)] = k[src];
                    hot[hot_offset(p, l, 1, g, (int)(t % bt), d, L, Hkv, D, bt)] = v[src];
                }
    }
    return 0;
}

/* splitmix64: advance the state by the golden gamma, return its mix. */
uint64_t oracle_splitmix64(uint64_t *state)
{
    uint64_t z = (*state += 0x9E3779B97F4A7C15ULL);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* Fisher-Yates over list[0..n): for i = n-1 down to 1 swap list[i] with
 * list[j], j = floor(r * (i + 1) / 2^64) for the next splitmix64 output r. */
void oracle_shuffle(int32_t *list, int64_t n, uint64_t seed)
{
    uint64_t st = seed;
    for (int64_t i = n - 1; i > 0; --i) {
        uint64_t r = oracle_splitmix64(&st);
        int64_t j = (int64_t)(((unsigned __int128)r * (uint64_t)(i + 1)) >> 64);
        int32_t tmp = list[i];
        list[i] = list[j];
        list[j] = tmp;
    }
}

/* Initial free list of a pool: 0..n-1 shuffled with the pool's seed. */
void oracle_free_list_init(int32_t *list, int64_t n, uint64_t seed)
{
    for (int64_t i = 0; i < n; ++i)
        list[i] = (int32_t)i;
    oracle_shuffle(list, n, seed);
}

/* Pop `count` blocks from the end of the free list into out[0..count), the
 * first popped going to logical block 0. Returns the new length or -1. */
int64_t oracle_free_list_pop(int32_t *list, int64_t n, int64_t count, int32_t *out)
{
    if (count > n)
        return -1;
    for (int64_t i = 0; i < count; ++i)
        out[i] = list[n - 1 - i];
    return n - count;
}

/* Push freed blocks back in logical order; returns the new length. */
int64_t oracle_free_list_push(int32_t *list, int64_t n, const int32_t *blocks, int64_t count)
{
    for (int64_t i = 0; i < count; ++i)
        list[n + i] = blocks[i];
    return n + count;
}
