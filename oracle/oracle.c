/*
 * oracle.c -- plain, slow CPU oracle for the Autoverse batched environment
 * step (Earle & Togelius, "Autoverse: an Evolvable Game Language for Learning
 * Robust Embodied Agents", arXiv 2407.04221).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg load this file's library.  It shares no code,
 * header, table or helper with the CUDA library; the only common inputs are
 * the packed rule records and thresholds made by the seeded generator.
 *
 * What it computes, and where it comes from:
 *
 *  - A board D is an H x W grid of multi-hot cells: bit c of a cell is tile
 *    channel c (Sec. 2.1 "one-hot encoded over the number of tile types";
 *    Sec. 2.2.1 calls the map "multi-hot"; a cell is a bitmask here).
 *  - A rewrite rule is an input patch I, an output patch O and a reward
 *    (Sec. 2.1; Fig. 2a caption).  Its effect on one patch C_t is the
 *    per-patch definition (Sec. 2.1, second displayed equation):
 *        C_{t+1} = O  if the input pattern is present in C_t,  else C_t.
 *    Input entries are ternary per (position, channel): present, absent or
 *    don't-care; "present" is the +1 weight of the matching convolution K_I
 *    (Sec. 2.1, first displayed equation), "absent" a -1 weight, so the test
 *    is still ReLU(conv - #present + 1) == 1.  Output entries are set, clear
 *    or unchanged per (position, tile channel).
 *  - The player acts by placing an invisible "force" tile next to itself
 *    (Sec. 2.1, movement paragraph).  Force is channel C: present during the
 *    step, never stored.
 *  - All rules apply in parallel to the same board D_t (Sec. 2.1, last
 *    paragraph of "Possible extensions"), so rule order does not matter.
 *  - A rule earns its reward each time it applies (Sec. 2.2.1, food rule).
 *
 * Readings where the paper is silent (each one is listed with its reason in
 * the design notes):
 *  - every rule is matched in its 4 rotations (0, 90, 180, 270 degrees
 *    counter-clockwise); each (rule, rotation, anchor) match counts once;
 *  - VALID anchors only: the whole window lies inside the grid;
 *  - conflicting writes: a bit changes if any match asks for the change:
 *        next = (F & ~CLR) | (~F & SET), force dropped;
 *  - actions: 0 no-op, 1 up (-y), 2 right (+x), 3 down (+y), 4 left (-x);
 *    values >= 5 act as no-op;
 *  - done when no goal tile is left, or the step counter reaches max_steps;
 *    with auto-reset the env returns its own initial map and t = 0.
 *
 * Integer-only counter RNG (SplitMix64 finaliser, Vigna, splitmix64.c):
 *   draw(seed, stream, a, b, c) =
 *       mix(mix(mix(seed + 0x9E3779B97F4A7C15*(stream+1)) ^ a) ^ (b<<32 | c))
 *
 * State hash: FNV-1a 64 (Fowler/Noll/Vo), offset basis 0xcbf29ce484222325,
 * prime 0x100000001b3, over the canonical grid bytes (row-major cells, each
 * cell little-endian in 1 byte if C <= 8 else 2 bytes, tile bits only).
 */
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_MAXSIDE 256
#define OR_MAXCELLS (OR_MAXSIDE * OR_MAXSIDE)
#define OR_MAXPAT 5
#define OR_RULE_BYTES 408

/* Oracle's own copy of the configuration (laid out like the generator's
 * config fields; every field is a 32-bit int). */
typedef struct {
    int32_t batch, H, W, C, n_rules, rules_per_env, max_steps, auto_reset;
    int32_t ch_player, ch_goal, ch_empty, ch_wall, border_wall, cum_per_env;
} or_cfg;

typedef struct {
    int h, w;
    int32_t reward;
    uint32_t present[25], absent[25], set[25], clear[25];
} or_pattern;

/* ------------------------------------------------------------------ RNG */
static uint64_t mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

uint64_t or_mix64(uint64_t z) { return mix64(z); }

uint64_t or_draw(uint64_t seed, uint64_t stream, uint64_t a, uint64_t b, uint64_t c)
{
    uint64_t z = mix64(seed + 0x9E3779B97F4A7C15ULL * (stream + 1));
    z = mix64(z ^ a);
    return mix64(z ^ ((b << 32) | c));
}

static uint32_t uniform_below(uint64_t d, uint32_t n)
{
    return (uint32_t)(((d >> 32) * (uint64_t)n) >> 32);
}

/* ------------------------------------------------------------------ hash */
uint64_t or_fnv1a64(const uint8_t *bytes, int64_t n)
{
    uint64_t h = 0xcbf29ce484222325ULL;
    for (int64_t i = 0; i < n; i++) {
        h ^= bytes[i];
        h *= 0x100000001b3ULL;
    }
    return h;
}

static int cell_bytes(int C) { return C <= 8 ? 1 : 2; }

static uint64_t hash_cells(const uint32_t *cells, int H, int W, int C)
{
    uint8_t buf[OR_MAXCELLS * 2];
    int nb = cell_bytes(C), n = 0;
    uint32_t tiles = (1u << C) - 1u;
    for (int p = 0; p < H * W; p++) {
        uint32_t v = cells[p] & tiles;
        buf[n++] = (uint8_t)(v & 0xff);
        if (nb == 2)
            buf[n++] = (uint8_t)(v >> 8);
    }
    return or_fnv1a64(buf, n);
}

/* ------------------------------------------------------- grid byte I/O */
static void load_grid(const void *src, int H, int W, int C, uint32_t *cells)
{
    const uint8_t *b = (const uint8_t *)src;
    for (int p = 0; p < H * W; p++)
        cells[p] = cell_bytes(C) == 1 ? b[p] : (uint32_t)b[2 * p] | ((uint32_t)b[2 * p + 1] << 8);
}

static void store_grid(const uint32_t *cells, int H, int W, int C, void *dst)
{
    uint8_t *b = (uint8_t *)dst;
    uint32_t tiles = (1u << C) - 1u;
    for (int p = 0; p < H * W; p++) {
        uint32_t v = cells[p] & tiles;
        if (cell_bytes(C) == 1) {
            b[p] = (uint8_t)v;
        } else {
            b[2 * p] = (uint8_t)(v & 0xff);
            b[2 * p + 1] = (uint8_t)(v >> 8);
        }
    }
}

uint64_t or_grid_hash(const void *grid, int H, int W, int C)
{
    uint32_t cells[OR_MAXCELLS];
    load_grid(grid, H, W, C, cells);
    return hash_cells(cells, H, W, C);
}

/* ------------------------------------------------------------- patterns */
static uint32_t rd32(const uint8_t *p)
{
    return (uint32_t)p[0] | ((uint32_t)p[1] << 8) | ((uint32_t)p[2] << 16) | ((uint32_t)p[3] << 24);
}

/* Parse one packed 408-byte record (little-endian). */
static void parse_rule(const uint8_t *rec, or_pattern *r)
{
    r->h = rec[0];
    r->w = rec[1];
    r->reward = (int32_t)rd32(rec + 4);
    for (int e = 0; e < 25; e++) {
        r->present[e] = rd32(rec + 8 + 4 * e);
        r->absent[e] = rd32(rec + 108 + 4 * e);
        r->set[e] = rd32(rec + 208 + 4 * e);
        r->clear[e] = rd32(rec + 308 + 4 * e);
    }
}

/* Rotate a pattern 90 degrees counter-clockwise: entry (i, k) of an h x w
 * pattern goes to (w-1-k, i) of the w x h result.  Input and output patterns
 * turn together; channels are not touched. */
static void rot90ccw(const or_pattern *in, or_pattern *out)
{
    or_pattern t;
    t.h = in->w;
    t.w = in->h;
    t.reward = in->reward;
    for (int i = 0; i < in->h; i++)
        for (int k = 0; k < in->w; k++) {
            int src = i * in->w + k;
            int dst = (in->w - 1 - k) * t.w + i;
            t.present[dst] = in->present[src];
            t.absent[dst] = in->absent[src];
            t.set[dst] = in->set[src];
            t.clear[dst] = in->clear[src];
        }
    *out = t;
}

static void rotated(const or_pattern *base, int j, or_pattern *out)
{
    *out = *base;
    for (int q = 0; q < j; q++)
        rot90ccw(out, out);
}

/* Exposed for tests: rotation j of one packed record. */
void or_rotate(const uint8_t *rec, int j, int32_t *hw, uint32_t *present, uint32_t *absent,
               uint32_t *set, uint32_t *clear)
{
    or_pattern b, r;
    parse_rule(rec, &b);
    rotated(&b, j, &r);
    hw[0] = r.h;
    hw[1] = r.w;
    for (int e = 0; e < r.h * r.w; e++) {
        present[e] = r.present[e];
        absent[e] = r.absent[e];
        set[e] = r.set[e];
        clear[e] = r.clear[e];
    }
}

/* ------------------------------------------------------------ one step */
static const int DY[5] = {0, -1, 0, 1, 0};
static const int DX[5] = {0, 0, 1, 0, -1};

typedef struct {
    const or_cfg *cfg;
    or_pattern rot[4 * 64]; /* rotation j of rule r at index 4r+j; R <= 64 */
    int R;
} or_rules;

static int load_rules(const or_cfg *cfg, const uint8_t *rules, int env, or_rules *out)
{
    int tab = cfg->rules_per_env ? env : 0;
    if (cfg->n_rules > 64)
        return -1;
    out->cfg = cfg;
    out->R = cfg->n_rules;
    for (int r = 0; r < cfg->n_rules; r++) {
        or_pattern base;
        parse_rule(rules + ((size_t)tab * cfg->n_rules + r) * OR_RULE_BYTES, &base);
        for (int j = 0; j < 4; j++)
            rotated(&base, j, &out->rot[4 * r + j]);
    }
    return 0;
}

/* The transition of the tile bits only (steps 1-4 of the documented
 * algorithm): force, match every rule rotation at every VALID anchor by
 * literal per-cell, per-channel comparison, then combine. */
static void transition(const or_cfg *cfg, const or_rules *rs, const uint32_t *G, int action,
                       uint32_t *N, int32_t *reward)
{
    const int H = cfg->H, W = cfg->W, C = cfg->C;
    uint32_t F[OR_MAXCELLS], SETm[OR_MAXCELLS], CLRm[OR_MAXCELLS];
    int32_t rew = 0;

    /* 1. force: next to every player cell, in the action's direction */
    for (int p = 0; p < H * W; p++)
        F[p] = G[p];
    if (action < 0 || action > 4)
        action = 0;
    if (cfg->ch_player >= 0 && action != 0) {
        for (int y = 0; y < H; y++)
            for (int x = 0; x < W; x++) {
                if (!((G[y * W + x] >> cfg->ch_player) & 1u))
                    continue;
                int yy = y + DY[action], xx = x + DX[action];
                if (yy >= 0 && yy < H && xx >= 0 && xx < W)
                    F[yy * W + xx] |= 1u << C;
            }
    }

    /* 2. accumulators */
    for (int p = 0; p < H * W; p++)
        SETm[p] = CLRm[p] = 0;

    /* 3. match: eq. 2 per patch, for every rule, rotation and anchor */
    for (int q = 0; q < 4 * rs->R; q++) {
        const or_pattern *P = &rs->rot[q];
        for (int y0 = 0; y0 + P->h <= H; y0++)
            for (int x0 = 0; x0 + P->w <= W; x0++) {
                int ok = 1;
                for (int i = 0; i < P->h && ok; i++)
                    for (int k = 0; k < P->w && ok; k++) {
                        uint32_t cell = F[(y0 + i) * W + (x0 + k)];
                        int e = i * P->w + k;
                        for (int c = 0; c <= C && ok; c++) {
                            uint32_t bit = (cell >> c) & 1u;
                            if (((P->present[e] >> c) & 1u) && !bit)
                                ok = 0;
                            if (((P->absent[e] >> c) & 1u) && bit)
                                ok = 0;
                        }
                    }
                if (!ok)
                    continue;
                rew += P->reward;
                for (int i = 0; i < P->h; i++)
                    for (int k = 0; k < P->w; k++) {
                        int e = i * P->w + k;
                        SETm[(y0 + i) * W + (x0 + k)] |= P->set[e];
                        CLRm[(y0 + i) * W + (x0 + k)] |= P->clear[e];
                    }
            }
    }

    /* 4. combine: a bit changes if any match asks for the change */
    uint32_t tiles = (1u << C) - 1u;
    for (int p = 0; p < H * W; p++)
        N[p] = ((F[p] & ~CLRm[p]) | (~F[p] & SETm[p])) & tiles;
    *reward = rew;
}

/* ----------------------------------------------------- variant semantics
 * The possible extensions at the end of Sec. 2.1: a rule may be applied only
 * once or a fixed number of times per step, the tiles to rewrite chosen by
 * taking the maximum over an additional channel of ordered or random index
 * values; and masking may let certain rules inhibit others.
 *
 * Readings (the paper only sketches them):
 *  - a match is (rule r, rotation j, anchor cell q = y0*W + x0); its key is
 *    (q << 2) | j with ordered indices, or ((draw(key_seed, 13, env, t, q)
 *    >> 48) << 14) | (q << 2) | j with random ones (t: the env's step counter
 *    before the step), so every match of a rule has a distinct key;
 *  - limit[r] = k > 0: of rule r's matches this step only the k with the
 *    largest keys apply (write and pay); 0: all apply;
 *  - inhibit[r]: when rule r has at least one match this step (before any
 *    limit or inhibition), every rule s with bit s of inhibit[r] set is
 *    suppressed this step (no writes, no reward) -- decided on raw matches,
 *    so the result does not depend on rule order. */
typedef struct {
    int32_t random_keys;
    int32_t _pad;
    uint64_t key_seed;
    int32_t limit[64];
    uint64_t inhibit[64];
} or_variant;

typedef struct {
    uint32_t key;
    int16_t j, y0, x0;
} or_match;

static int cmp_match_desc(const void *a, const void *b)
{
    uint32_t ka = ((const or_match *)a)->key, kb = ((const or_match *)b)->key;
    return ka < kb ? 1 : ka > kb ? -1 : 0;
}

static void transition_variant(const or_cfg *cfg, const or_rules *rs, const or_variant *v, uint64_t env,
                               int32_t t, const uint32_t *G, int action, uint32_t *N, int32_t *reward,
                               or_match *buf)
{
    const int H = cfg->H, W = cfg->W, C = cfg->C;
    uint32_t F[OR_MAXCELLS], SETm[OR_MAXCELLS], CLRm[OR_MAXCELLS];
    int32_t rew = 0;
    for (int p = 0; p < H * W; p++)
        F[p] = G[p];
    if (action < 0 || action > 4)
        action = 0;
    if (cfg->ch_player >= 0 && action != 0)
        for (int y = 0; y < H; y++)
            for (int x = 0; x < W; x++) {
                if (!((G[y * W + x] >> cfg->ch_player) & 1u))
                    continue;
                int yy = y + DY[action], xx = x + DX[action];
                if (yy >= 0 && yy < H && xx >= 0 && xx < W)
                    F[yy * W + xx] |= 1u << C;
            }
    for (int p = 0; p < H * W; p++)
        SETm[p] = CLRm[p] = 0;

    /* raw matches of every rule, before limits and inhibition */
    int count[64];
    int start[65];
    start[0] = 0;
    for (int r = 0; r < rs->R; r++) {
        int n = 0;
        for (int j = 0; j < 4; j++) {
            const or_pattern *P = &rs->rot[4 * r + j];
            for (int y0 = 0; y0 + P->h <= H; y0++)
                for (int x0 = 0; x0 + P->w <= W; x0++) {
                    int ok = 1;
                    for (int i = 0; i < P->h && ok; i++)
                        for (int k = 0; k < P->w && ok; k++) {
                            uint32_t cell = F[(y0 + i) * W + (x0 + k)];
                            int e = i * P->w + k;
                            for (int c = 0; c <= C && ok; c++) {
                                uint32_t bit = (cell >> c) & 1u;
                                if (((P->present[e] >> c) & 1u) && !bit)
                                    ok = 0;
                                if (((P->absent[e] >> c) & 1u) && bit)
                                    ok = 0;
                            }
                        }
                    if (!ok)
                        continue;
                    const uint32_t q = (uint32_t)(y0 * W + x0);
                    uint32_t key = (q << 2) | (uint32_t)j;
                    if (v->random_keys)
                        key |= (uint32_t)(or_draw(v->key_seed, 13, env, (uint64_t)(uint32_t)t, q) >> 48) << 14;
                    or_match *m = &buf[start[r] + n++];
                    m->key = key;
                    m->j = (int16_t)j;
                    m->y0 = (int16_t)y0;
                    m->x0 = (int16_t)x0;
                }
        }
        count[r] = n;
        start[r + 1] = start[r] + n;
    }
    /* inhibition, from raw matches */
    uint64_t suppressed = 0;
    for (int r = 0; r < rs->R; r++)
        if (count[r] > 0)
            suppressed |= v->inhibit[r];
    /* the applied matches: all, or the limit[r] with the largest keys */
    for (int r = 0; r < rs->R; r++) {
        if ((suppressed >> r) & 1u)
            continue;
        or_match *list = &buf[start[r]];
        int n = count[r];
        if (v->limit[r] > 0 && n > v->limit[r]) {
            qsort(list, (size_t)n, sizeof(or_match), cmp_match_desc);
            n = v->limit[r];
        }
        for (int m = 0; m < n; m++) {
            const or_pattern *P = &rs->rot[4 * r + list[m].j];
            rew += P->reward;
            for (int i = 0; i < P->h; i++)
                for (int k = 0; k < P->w; k++) {
                    int e = i * P->w + k;
                    SETm[(list[m].y0 + i) * W + (list[m].x0 + k)] |= P->set[e];
                    CLRm[(list[m].y0 + i) * W + (list[m].x0 + k)] |= P->clear[e];
                }
        }
    }
    uint32_t tiles = (1u << C) - 1u;
    for (int p = 0; p < H * W; p++)
        N[p] = ((F[p] & ~CLRm[p]) | (~F[p] & SETm[p])) & tiles;
    *reward = rew;
}

/* Room for every raw match of one step: 4 rotations x H*W anchors x R rules. */
static or_match *match_buffer(const or_cfg *cfg)
{
    return (or_match *)malloc(sizeof(or_match) * 4 * (size_t)cfg->H * cfg->W * (cfg->n_rules > 0 ? cfg->n_rules : 1));
}

static int goal_left(const or_cfg *cfg, const uint32_t *N)
{
    if (cfg->ch_goal < 0)
        return 1;
    for (int p = 0; p < cfg->H * cfg->W; p++)
        if ((N[p] >> cfg->ch_goal) & 1u)
            return 1;
    return 0;
}

/* Steps 5-6: done and auto-reset.  *t is the env's step counter. */
static uint8_t finish(const or_cfg *cfg, uint32_t *N, const uint32_t *init, int32_t *t)
{
    *t += 1;
    int done = !goal_left(cfg, N) || (cfg->max_steps > 0 && *t >= cfg->max_steps);
    if (done && cfg->auto_reset) {
        for (int p = 0; p < cfg->H * cfg->W; p++)
            N[p] = init[p];
        *t = 0;
    }
    return (uint8_t)done;
}

/* ---------------------------------------------------------------- reset */
int or_reset(const or_cfg *cfg, const uint32_t *cum_all, uint64_t seed, int env, void *grid_out)
{
    const int H = cfg->H, W = cfg->W, C = cfg->C;
    const uint32_t *cum = cum_all + (size_t)(cfg->cum_per_env ? env : 0) * C;
    uint32_t cells[OR_MAXCELLS];
    for (int y = 0; y < H; y++)
        for (int x = 0; x < W; x++) {
            int border = y == 0 || y == H - 1 || x == 0 || x == W - 1;
            uint32_t v;
            if (cfg->border_wall && border) {
                v = cfg->ch_wall >= 0 ? 1u << cfg->ch_wall : 0u;
            } else {
                uint32_t u = (uint32_t)(or_draw(seed, 1, (uint64_t)env, (uint64_t)y, (uint64_t)x) >> 40);
                int t = 0;
                while (t < C - 1 && !(u < cum[t]))
                    t++;
                v = 1u << t;
            }
            cells[y * W + x] = v;
        }
    if (cfg->ch_player >= 0) {
        uint64_t d = or_draw(seed, 2, (uint64_t)env, 0, 0);
        int n_empty = 0;
        if (cfg->ch_empty >= 0)
            for (int p = 0; p < H * W; p++)
                n_empty += (cells[p] >> cfg->ch_empty) & 1u;
        int chosen = -1;
        if (n_empty > 0) {
            uint32_t k = uniform_below(d, (uint32_t)n_empty);
            for (int p = 0, seen = 0; p < H * W; p++)
                if ((cells[p] >> cfg->ch_empty) & 1u) {
                    if (seen == (int)k) {
                        chosen = p;
                        break;
                    }
                    seen++;
                }
        } else {
            int n_int = 0;
            for (int y = 0; y < H; y++)
                for (int x = 0; x < W; x++) {
                    int border = y == 0 || y == H - 1 || x == 0 || x == W - 1;
                    n_int += !(cfg->border_wall && border);
                }
            if (n_int > 0) {
                uint32_t k = uniform_below(d, (uint32_t)n_int);
                for (int y = 0, seen = 0; y < H && chosen < 0; y++)
                    for (int x = 0; x < W; x++) {
                        int border = y == 0 || y == H - 1 || x == 0 || x == W - 1;
                        if (cfg->border_wall && border)
                            continue;
                        if (seen == (int)k) {
                            chosen = y * W + x;
                            break;
                        }
                        seen++;
                    }
            }
        }
        if (chosen >= 0)
            cells[chosen] |= 1u << cfg->ch_player;
    }
    store_grid(cells, H, W, C, grid_out);
    return 0;
}

/* ------------------------------------------------------------ threading */
typedef struct {
    int n, threads;
    void *ctx;
    int (*fn)(void *ctx, int item);
    int next, err;
    pthread_mutex_t mu;
} pool;

static void *pool_worker(void *arg)
{
    pool *p = (pool *)arg;
    for (;;) {
        pthread_mutex_lock(&p->mu);
        int item = p->next++;
        pthread_mutex_unlock(&p->mu);
        if (item >= p->n)
            break;
        int e = p->fn(p->ctx, item);
        if (e) {
            pthread_mutex_lock(&p->mu);
            p->err = e;
            pthread_mutex_unlock(&p->mu);
        }
    }
    return NULL;
}

static int run_pool(int n, int threads, void *ctx, int (*fn)(void *, int))
{
    pool p = {n, threads, ctx, fn, 0, 0};
    pthread_mutex_init(&p.mu, NULL);
    if (threads < 1 || n <= 1)
        threads = 1;
    if (threads > 256)
        threads = 256;
    /* Workers get large stacks: a 256 x 256 board puts several whole-board
     * arrays on the stack of each step. */
    pthread_attr_t attr;
    pthread_attr_init(&attr);
    pthread_attr_setstacksize(&attr, (size_t)64 << 20);
    pthread_t tid[256];
    int started = 0;
    for (int i = 0; i < threads; i++)
        if (pthread_create(&tid[i], &attr, pool_worker, &p) == 0)
            started++;
        else
            break;
    pthread_attr_destroy(&attr);
    if (started == 0)
        pool_worker(&p);
    for (int i = 0; i < started; i++)
        pthread_join(tid[i], NULL);
    pthread_mutex_destroy(&p.mu);
    return p.err;
}

static int check_cfg(const or_cfg *c)
{
    if (c->H < 1 || c->W < 1 || c->H > OR_MAXSIDE || c->W > OR_MAXSIDE || c->C < 1 || c->C > 16 ||
        c->n_rules < 0 || c->n_rules > 64)
        return -1;
    return 0;
}

static size_t grid_bytes(const or_cfg *c) { return (size_t)c->H * c->W * cell_bytes(c->C); }

/* ------------------------------------------------------- batched step */
typedef struct {
    const or_cfg *cfg;
    const uint8_t *rules;
    const int32_t *env_ids;
    const uint8_t *grids_in, *inits;
    const int32_t *t_in;
    const uint8_t *actions;
    uint8_t *grids_out;
    int32_t *t_out, *rewards;
    uint8_t *dones;
    const or_variant *v; /* NULL: standard semantics */
} step_job;

static int step_item(void *ctx, int n)
{
    step_job *j = (step_job *)ctx;
    const or_cfg *cfg = j->cfg;
    or_rules *rs = (or_rules *)malloc(sizeof(or_rules));
    if (!rs)
        return -2;
    int env = j->env_ids ? j->env_ids[n] : n;
    if (load_rules(cfg, j->rules, env, rs)) {
        free(rs);
        return -1;
    }
    uint32_t G[OR_MAXCELLS], I[OR_MAXCELLS], N[OR_MAXCELLS];
    size_t gb = grid_bytes(cfg);
    load_grid(j->grids_in + gb * n, cfg->H, cfg->W, cfg->C, G);
    load_grid(j->inits + gb * n, cfg->H, cfg->W, cfg->C, I);
    int32_t rew, t = j->t_in[n];
    if (j->v) {
        or_match *buf = match_buffer(cfg);
        if (!buf) {
            free(rs);
            return -2;
        }
        transition_variant(cfg, rs, j->v, (uint64_t)env, t, G, j->actions[n], N, &rew, buf);
        free(buf);
    } else {
        transition(cfg, rs, G, j->actions[n], N, &rew);
    }
    j->dones[n] = finish(cfg, N, I, &t);
    j->rewards[n] = rew;
    j->t_out[n] = t;
    store_grid(N, cfg->H, cfg->W, cfg->C, j->grids_out + gb * n);
    free(rs);
    return 0;
}

/* One step of n envs.  env_ids (nullable) maps item n to the env index that
 * selects its rule table; grids are canonical [n][H][W] cell words. */
int or_step_batch_v(const or_cfg *cfg, const uint8_t *rules, const or_variant *v, int n,
                    const int32_t *env_ids, const void *grids_in, const void *inits,
                    const int32_t *t_in, const uint8_t *actions, void *grids_out, int32_t *t_out,
                    int32_t *rewards, uint8_t *dones, int threads)
{
    if (check_cfg(cfg))
        return -1;
    step_job j = {cfg, rules, env_ids, (const uint8_t *)grids_in, (const uint8_t *)inits, t_in,
                  actions, (uint8_t *)grids_out, t_out, rewards, dones, v};
    return run_pool(n, threads, &j, step_item);
}

int or_step_batch(const or_cfg *cfg, const uint8_t *rules, int n, const int32_t *env_ids,
                  const void *grids_in, const void *inits, const int32_t *t_in,
                  const uint8_t *actions, void *grids_out, int32_t *t_out, int32_t *rewards,
                  uint8_t *dones, int threads)
{
    return or_step_batch_v(cfg, rules, NULL, n, env_ids, grids_in, inits, t_in, actions, grids_out,
                           t_out, rewards, dones, threads);
}

/* -------------------------------------------------------------- rollout */
typedef struct {
    const or_cfg *cfg;
    const uint8_t *rules;
    const int32_t *env_ids;
    int n, n_steps;
    uint64_t action_seed;
    uint8_t *grids;
    const uint8_t *inits;
    int32_t *t;
    uint8_t *obs_traj;
    int32_t *rew_traj;
    uint8_t *done_traj;
    int32_t *rew_sum;
    const or_variant *v; /* NULL: standard semantics */
} roll_job;

static int roll_item(void *ctx, int n)
{
    roll_job *j = (roll_job *)ctx;
    const or_cfg *cfg = j->cfg;
    or_rules *rs = (or_rules *)malloc(sizeof(or_rules));
    if (!rs)
        return -2;
    int env = j->env_ids ? j->env_ids[n] : n;
    if (load_rules(cfg, j->rules, env, rs)) {
        free(rs);
        return -1;
    }
    uint32_t G[OR_MAXCELLS], I[OR_MAXCELLS], N[OR_MAXCELLS];
    size_t gb = grid_bytes(cfg);
    load_grid(j->grids + gb * n, cfg->H, cfg->W, cfg->C, G);
    load_grid(j->inits + gb * n, cfg->H, cfg->W, cfg->C, I);
    int32_t t = j->t[n], sum = 0;
    or_match *buf = NULL;
    if (j->v && !(buf = match_buffer(cfg))) {
        free(rs);
        return -2;
    }
    for (int s = 0; s < j->n_steps; s++) {
        int a = (int)uniform_below(or_draw(j->action_seed, 4, (uint64_t)env, 0, (uint64_t)s), 5);
        int32_t rew;
        if (j->v)
            transition_variant(cfg, rs, j->v, (uint64_t)env, t, G, a, N, &rew, buf);
        else
            transition(cfg, rs, G, a, N, &rew);
        uint8_t d = finish(cfg, N, I, &t);
        sum += rew;
        size_t slot = (size_t)s * j->n + n;
        if (j->obs_traj)
            store_grid(N, cfg->H, cfg->W, cfg->C, j->obs_traj + gb * slot);
        if (j->rew_traj)
            j->rew_traj[slot] = rew;
        if (j->done_traj)
            j->done_traj[slot] = d;
        memcpy(G, N, sizeof(uint32_t) * cfg->H * cfg->W);
    }
    store_grid(G, cfg->H, cfg->W, cfg->C, j->grids + gb * n);
    j->t[n] = t;
    if (j->rew_sum)
        j->rew_sum[n] = sum;
    free(buf);
    free(rs);
    return 0;
}

/* n_steps fused steps of n envs with on-the-fly actions
 * a = uniform5(draw(action_seed, 4, env, 0, s)).  grids and t are updated in
 * place; trajectories are [n_steps][n] (nullable). */
int or_rollout_v(const or_cfg *cfg, const uint8_t *rules, const or_variant *v, int n,
                 const int32_t *env_ids, void *grids, const void *inits, int32_t *t, int n_steps,
                 uint64_t action_seed, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj,
                 int32_t *rew_sum, int threads)
{
    if (check_cfg(cfg) || n_steps < 0)
        return -1;
    roll_job j = {cfg, rules, env_ids, n, n_steps, action_seed, (uint8_t *)grids,
                  (const uint8_t *)inits, t, (uint8_t *)obs_traj, rew_traj, done_traj, rew_sum, v};
    return run_pool(n, threads, &j, roll_item);
}

int or_rollout(const or_cfg *cfg, const uint8_t *rules, int n, const int32_t *env_ids, void *grids,
               const void *inits, int32_t *t, int n_steps, uint64_t action_seed, void *obs_traj,
               int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, int threads)
{
    return or_rollout_v(cfg, rules, NULL, n, env_ids, grids, inits, t, n_steps, action_seed,
                        obs_traj, rew_traj, done_traj, rew_sum, threads);
}

/* --------------------------------------------------------------- expand */
typedef struct {
    const or_cfg *cfg;
    const uint8_t *rules;
    const int32_t *env_ids;
    int F;
    const uint8_t *parents;
    uint8_t *children;
    int32_t *rewards;
    uint8_t *done;
    uint64_t *hashes;
} exp_job;

static int expand_item(void *ctx, int n)
{
    exp_job *j = (exp_job *)ctx;
    const or_cfg *cfg = j->cfg;
    or_rules *rs = (or_rules *)malloc(sizeof(or_rules));
    if (!rs)
        return -2;
    int env = j->env_ids ? j->env_ids[n] : n;
    if (load_rules(cfg, j->rules, env, rs)) {
        free(rs);
        return -1;
    }
    size_t gb = grid_bytes(cfg);
    uint32_t G[OR_MAXCELLS], N[OR_MAXCELLS];
    for (int f = 0; f < j->F; f++) {
        load_grid(j->parents + gb * ((size_t)n * j->F + f), cfg->H, cfg->W, cfg->C, G);
        for (int a = 0; a < 5; a++) {
            size_t slot = ((size_t)n * j->F + f) * 5 + a;
            int32_t rew;
            transition(cfg, rs, G, a, N, &rew);
            j->rewards[slot] = rew;
            if (j->done)
                j->done[slot] = (uint8_t)!goal_left(cfg, N);
            j->hashes[slot] = hash_cells(N, cfg->H, cfg->W, cfg->C);
            store_grid(N, cfg->H, cfg->W, cfg->C, j->children + gb * slot);
        }
    }
    free(rs);
    return 0;
}

/* Every parent [n][F] stepped by all 5 actions -> children [n][F][5], their
 * rewards, done flags (goal exhausted) and FNV-1a hashes.  No step counter
 * and no reset: a child is the raw transition. */
int or_expand(const or_cfg *cfg, const uint8_t *rules, int n, const int32_t *env_ids,
              const void *parents, int F, void *children, int32_t *rewards, uint8_t *done,
              uint64_t *hashes, int threads)
{
    if (check_cfg(cfg) || F < 0)
        return -1;
    exp_job j = {cfg, rules, env_ids, F, (const uint8_t *)parents, (uint8_t *)children, rewards,
                 done, hashes};
    return run_pool(n, threads, &j, expand_item);
}

/* --------------------------------------------------------------- search */
typedef struct {
    int32_t cum;
    uint64_t hash;
    int idx; /* candidate index f*5+a: ties in dedup keep the smallest */
    uint8_t done;
} cand;

static int cmp_hash_then_best(const void *a, const void *b)
{
    const cand *x = (const cand *)a, *y = (const cand *)b;
    if (x->hash != y->hash)
        return x->hash < y->hash ? -1 : 1;
    if (x->cum != y->cum)
        return x->cum > y->cum ? -1 : 1;
    return x->idx < y->idx ? -1 : (x->idx > y->idx);
}

static int cmp_rank(const void *a, const void *b)
{
    const cand *x = (const cand *)a, *y = (const cand *)b;
    if (x->cum != y->cum)
        return x->cum > y->cum ? -1 : 1;
    if (x->hash != y->hash)
        return x->hash < y->hash ? -1 : 1;
    return 0;
}

static int cmp_u64(const void *a, const void *b)
{
    uint64_t x = *(const uint64_t *)a, y = *(const uint64_t *)b;
    return x < y ? -1 : (x > y);
}

typedef struct {
    const or_cfg *cfg;
    const uint8_t *rules;
    const int32_t *env_ids;
    int iterations, k;
    const uint8_t *roots;
    uint8_t *front_grids; /* [n][k] */
    int32_t *front_cum;
    uint64_t *front_hash;
    uint8_t *front_done;
    int32_t *n_front;   /* [n] */
    int32_t *trace_n;   /* [n][iterations] frontier size after each iteration */
    int32_t *trace_best;/* [n][iterations] best cum in that frontier (INT32_MIN if empty) */
    int32_t *n_visited; /* [n] */
} search_job;

static int search_item(void *ctx, int n)
{
    search_job *j = (search_job *)ctx;
    const or_cfg *cfg = j->cfg;
    const int HW = cfg->H * cfg->W, K = j->k;
    int env = j->env_ids ? j->env_ids[n] : n;
    int rc = -2;
    or_rules *rs = (or_rules *)malloc(sizeof(or_rules));
    uint32_t *front = (uint32_t *)malloc(sizeof(uint32_t) * HW * (size_t)K);
    uint32_t *kids = (uint32_t *)malloc(sizeof(uint32_t) * HW * (size_t)K * 5);
    uint32_t *next = (uint32_t *)malloc(sizeof(uint32_t) * HW * (size_t)K);
    int32_t *fcum = (int32_t *)malloc(sizeof(int32_t) * K), *ncum = (int32_t *)malloc(sizeof(int32_t) * K);
    uint64_t *fh = (uint64_t *)malloc(8 * (size_t)K), *nh = (uint64_t *)malloc(8 * (size_t)K);
    uint8_t *fd = (uint8_t *)malloc(K), *nd = (uint8_t *)malloc(K);
    cand *cs = (cand *)malloc(sizeof(cand) * (size_t)K * 5);
    size_t vcap = 1 + (size_t)K * j->iterations;
    uint64_t *vis = (uint64_t *)malloc(8 * vcap);
    if (!rs || !front || !kids || !next || !fcum || !ncum || !fh || !nh || !fd || !nd || !cs || !vis)
        goto out;
    rc = -1;
    if (load_rules(cfg, j->rules, env, rs))
        goto out;
    rc = 0;

    /* root: cum 0, visited = {hash(root)} */
    int nf = 1;
    load_grid(j->roots + (size_t)n * HW * cell_bytes(cfg->C), cfg->H, cfg->W, cfg->C, front);
    fcum[0] = 0;
    fh[0] = hash_cells(front, cfg->H, cfg->W, cfg->C);
    fd[0] = (uint8_t)!goal_left(cfg, front);
    size_t nv = 0;
    vis[nv++] = fh[0];

    for (int it = 0; it < j->iterations; it++) {
        /* expand every live frontier node by all 5 actions */
        int nc = 0;
        for (int f = 0; f < nf; f++) {
            if (fd[f])
                continue; /* done nodes are kept but not expanded */
            for (int a = 0; a < 5; a++) {
                int32_t rew;
                uint32_t *child = kids + (size_t)(f * 5 + a) * HW;
                transition(cfg, rs, front + (size_t)f * HW, a, child, &rew);
                cs[nc].cum = fcum[f] + rew;
                cs[nc].hash = hash_cells(child, cfg->H, cfg->W, cfg->C);
                cs[nc].idx = f * 5 + a;
                cs[nc].done = (uint8_t)!goal_left(cfg, child);
                nc++;
            }
        }
        /* drop states already visited (the shallower copy is kept) */
        int m = 0;
        for (int c = 0; c < nc; c++)
            if (!bsearch(&cs[c].hash, vis, nv, 8, cmp_u64))
                cs[m++] = cs[c];
        /* equal states: keep the highest cumulative reward */
        qsort(cs, m, sizeof(cand), cmp_hash_then_best);
        int u = 0;
        for (int c = 0; c < m; c++)
            if (c == 0 || cs[c].hash != cs[c - 1].hash)
                cs[u++] = cs[c];
        /* greedy: best cumulative reward first, ties by hash */
        qsort(cs, u, sizeof(cand), cmp_rank);
        int take = u < K ? u : K;
        for (int s = 0; s < take; s++) {
            memcpy(next + (size_t)s * HW, kids + (size_t)cs[s].idx * HW, sizeof(uint32_t) * HW);
            ncum[s] = cs[s].cum;
            nh[s] = cs[s].hash;
            nd[s] = cs[s].done;
            vis[nv++] = cs[s].hash;
        }
        qsort(vis, nv, 8, cmp_u64);
        memcpy(front, next, sizeof(uint32_t) * HW * (size_t)take);
        memcpy(fcum, ncum, sizeof(int32_t) * take);
        memcpy(fh, nh, 8 * (size_t)take);
        memcpy(fd, nd, take);
        nf = take;
        if (j->trace_n)
            j->trace_n[(size_t)n * j->iterations + it] = nf;
        if (j->trace_best)
            j->trace_best[(size_t)n * j->iterations + it] = nf ? fcum[0] : INT32_MIN;
    }
    size_t gb = (size_t)HW * cell_bytes(cfg->C);
    for (int f = 0; f < nf; f++) {
        store_grid(front + (size_t)f * HW, cfg->H, cfg->W, cfg->C,
                   j->front_grids + gb * ((size_t)n * K + f));
        j->front_cum[(size_t)n * K + f] = fcum[f];
        j->front_hash[(size_t)n * K + f] = fh[f];
        j->front_done[(size_t)n * K + f] = fd[f];
    }
    j->n_front[n] = nf;
    j->n_visited[n] = (int32_t)nv;
out:
    free(rs); free(front); free(kids); free(next); free(fcum); free(ncum);
    free(fh); free(nh); free(fd); free(nd); free(cs); free(vis);
    return rc;
}

/* Greedy best-first beam search from each root: `iterations` rounds of
 * expand-all-actions, drop visited, dedup, keep top-k by (cum desc, hash asc). */
int or_search(const or_cfg *cfg, const uint8_t *rules, int n, const int32_t *env_ids,
              const void *roots, int iterations, int k, void *front_grids, int32_t *front_cum,
              uint64_t *front_hash, uint8_t *front_done, int32_t *n_front, int32_t *trace_n,
              int32_t *trace_best, int32_t *n_visited, int threads)
{
    if (check_cfg(cfg) || iterations < 0 || k < 1)
        return -1;
    search_job j = {cfg, rules, env_ids, iterations, k, (const uint8_t *)roots,
                    (uint8_t *)front_grids, front_cum, front_hash, front_done, n_front, trace_n,
                    trace_best, n_visited};
    return run_pool(n, threads, &j, search_item);
}

/* ------------------------------------------------- policy observation
 * Sec. 3.2 (imitation learning): the agent observes a local patch of tiles
 * centred on the player's current position, together with a binary form of
 * the environment's rules.  Sec. 4, Table 1, varies the patch width (5, 10,
 * 20, 31) and pads the map with zeros where the patch leaves it; Table 2
 * hides the rules by putting zeros in their place.
 *
 * Readings (the paper says no more):
 *  - the player is the first cell in row-major order that holds the player
 *    bit; with no such cell every entry of the patch is 0;
 *  - patch entry (i, k) is board cell (py - window/2 + i, px - window/2 + k),
 *    integer division, so the player sits at (window/2, window/2) and a
 *    patch 2*max(H, W) - 1 wide holds the whole board wherever the player is;
 *  - cells outside the board read as 0 in every channel;
 *  - the patch is written channels-last as bytes [window][window][C]: byte c
 *    of an entry is tile bit c (force is never stored, so never observed).
 * player_yx (nullable) receives (py, px), or (-1, -1) without a player. */
int or_observe(const or_cfg *cfg, int n, const void *grids, int window, uint8_t *obs,
               int32_t *player_yx)
{
    if (check_cfg(cfg) || n < 0 || window < 1 || cfg->ch_player < 0 || cfg->ch_player >= cfg->C)
        return -1;
    const int H = cfg->H, W = cfg->W, C = cfg->C;
    uint32_t cells[OR_MAXCELLS];
    for (int b = 0; b < n; b++) {
        load_grid((const uint8_t *)grids + (size_t)b * grid_bytes(cfg), H, W, C, cells);
        int py = -1, px = -1;
        for (int q = 0; q < H * W && py < 0; q++)
            if ((cells[q] >> cfg->ch_player) & 1u) {
                py = q / W;
                px = q % W;
            }
        uint8_t *o = obs + (size_t)b * window * window * C;
        for (int i = 0; i < window; i++)
            for (int k = 0; k < window; k++) {
                int y = py - window / 2 + i, x = px - window / 2 + k;
                int on_board = py >= 0 && y >= 0 && y < H && x >= 0 && x < W;
                for (int c = 0; c < C; c++)
                    o[((size_t)i * window + k) * C + c] =
                        on_board ? (uint8_t)((cells[y * W + x] >> c) & 1u) : 0;
            }
        if (player_yx) {
            player_yx[2 * b] = py;
            player_yx[2 * b + 1] = px;
        }
    }
    return 0;
}

/* Binary form of the rules (Sec. 3.2).  Reading: every rule becomes four
 * binary planes over a 5 x 5 frame with C + 1 channels (force last):
 * plane 0 the present entries and plane 1 the absent entries of the input
 * pattern (the +1 and -1 weights of the matching kernel, Sec. 2.1), plane 2
 * the set entries and plane 3 the clear entries of the output pattern (tile
 * channels only, so their force channel is 0).  Entry (i, k) of the base,
 * unrotated h x w pattern sits at frame row i, column k; the rest of the
 * frame is 0.  bits: [n_tables][R][4][5][5][C+1]; reward (nullable):
 * [n_tables][R], the rule's reward as given. */
int or_rule_obs(const or_cfg *cfg, const uint8_t *rules, int n_tables, uint8_t *bits,
                int32_t *reward)
{
    if (check_cfg(cfg) || n_tables < 0)
        return -1;
    const int R = cfg->n_rules, NCH = cfg->C + 1;
    for (int t = 0; t < n_tables; t++)
        for (int r = 0; r < R; r++) {
            or_pattern p;
            parse_rule(rules + ((size_t)t * R + r) * OR_RULE_BYTES, &p);
            uint8_t *o = bits + ((size_t)t * R + r) * 4 * 25 * NCH;
            memset(o, 0, (size_t)4 * 25 * NCH);
            for (int i = 0; i < p.h; i++)
                for (int k = 0; k < p.w; k++) {
                    const int e = i * p.w + k, f = i * 5 + k;
                    for (int c = 0; c < NCH; c++) {
                        o[(0 * 25 + f) * NCH + c] = (p.present[e] >> c) & 1u;
                        o[(1 * 25 + f) * NCH + c] = (p.absent[e] >> c) & 1u;
                        o[(2 * 25 + f) * NCH + c] = c < cfg->C ? (p.set[e] >> c) & 1u : 0;
                        o[(3 * 25 + f) * NCH + c] = c < cfg->C ? (p.clear[e] >> c) & 1u : 0;
                    }
                }
            if (reward)
                reward[(size_t)t * R + r] = p.reward;
        }
    return 0;
}

/* ------------------------------------------------------------ mutation
 * The mutation operators of the evolution loop (Sec. 3.1.1):
 *  - the initial map, a multi-hot array, is mutated by flipping bits at
 *    random (last paragraph);
 *  - the mutable rules (the empty "no-op" rules added to the base game, not
 *    the base game's own) are mutated by changing tiles of the input and/or
 *    output pattern at various positions (first paragraph);
 *  - a rule's reward may be changed as well, to positive or negative values
 *    (second paragraph).
 *
 * Readings (the paper gives no rates, order or encoding):
 *  - every decision is an independent Bernoulli draw from the counter RNG,
 *    u = draw >> 40 (24 bits), taken when u < p (p in units of 2^-24);
 *  - map: bit c of cell q = y*W + x of env b flips when
 *    draw(seed, 9, b, q, c) >> 40 < p_map, for the channels in map_channels;
 *  - rules: an input entry (rule r, pattern entry e < h*w, channel c <= C)
 *    has three states, don't-care / present / absent, and an output entry
 *    (channel c < C) three, unchanged / set / clear; with d =
 *    draw(seed, 10 (input) or 11 (output), t, 25*r + e, c), the entry changes
 *    when d >> 40 < p_rule, to the next state (cyclically) when bit 39 of d
 *    is 0 and the one after it when 1 -- a change to one of the two other
 *    states, each equally likely;
 *  - reward: with d = draw(seed, 12, t, r, 0), when d >> 40 < p_reward the
 *    reward becomes reward_min + ((draw(seed, 12, t, r, 1) >> 32) * n >> 32),
 *    n = reward_max - reward_min + 1 (uniform, may equal the old one);
 *  - only rules whose bit is set in mutable_rules change; the pattern size
 *    h x w is kept.
 * env_ids (nullable) give the global environment / table index used in the
 * draws for each of the n maps and n tables passed. */
typedef struct {
    uint32_t p_map, map_channels, p_rule, p_reward;
    int32_t reward_min, reward_max;
    uint64_t mutable_rules;
} or_mutation;

static void wr32(uint8_t *p, uint32_t v)
{
    p[0] = (uint8_t)v;
    p[1] = (uint8_t)(v >> 8);
    p[2] = (uint8_t)(v >> 16);
    p[3] = (uint8_t)(v >> 24);
}

/* Ternary state of bit c in a pair of masks (one, two): 0 neither, 1 one, 2 two. */
static int tern_get(uint32_t one, uint32_t two, int c) { return ((one >> c) & 1u) ? 1 : ((two >> c) & 1u) ? 2 : 0; }

static void tern_set(uint32_t *one, uint32_t *two, int c, int state)
{
    *one &= ~(1u << c);
    *two &= ~(1u << c);
    if (state == 1)
        *one |= 1u << c;
    else if (state == 2)
        *two |= 1u << c;
}

static int mutated_state(uint64_t d, uint32_t p, int state)
{
    if ((uint32_t)(d >> 40) >= p)
        return state;
    return (state + 1 + (int)((d >> 39) & 1u)) % 3;
}

int or_mutate(int n, const int32_t *env_ids, int H, int W, int C, int R, const or_mutation *m,
              uint64_t seed, void *maps, uint8_t *rules)
{
    if (n < 0 || H < 1 || W < 1 || H > OR_MAXSIDE || W > OR_MAXSIDE || C < 1 || C > 16 || R < 0 ||
        R > 64)
        return -1;
    const size_t gb = (size_t)H * W * cell_bytes(C);
    uint32_t cells[OR_MAXCELLS];
    for (int i = 0; i < n; i++) {
        const uint64_t b = env_ids ? (uint64_t)env_ids[i] : (uint64_t)i;
        if (maps) {
            uint8_t *g = (uint8_t *)maps + (size_t)i * gb;
            load_grid(g, H, W, C, cells);
            for (int q = 0; q < H * W; q++)
                for (int c = 0; c < C; c++)
                    if (((m->map_channels >> c) & 1u) && (uint32_t)(or_draw(seed, 9, b, q, c) >> 40) < m->p_map)
                        cells[q] ^= 1u << c;
            store_grid(cells, H, W, C, g);
        }
        if (!rules)
            continue;
        for (int r = 0; r < R; r++) {
            if (!((m->mutable_rules >> r) & 1u))
                continue;
            uint8_t *rec = rules + ((size_t)i * R + r) * OR_RULE_BYTES;
            or_pattern p;
            parse_rule(rec, &p);
            for (int e = 0; e < p.h * p.w; e++) {
                for (int c = 0; c <= C; c++) {
                    const uint64_t d = or_draw(seed, 10, b, 25u * r + e, c);
                    tern_set(&p.present[e], &p.absent[e], c,
                             mutated_state(d, m->p_rule, tern_get(p.present[e], p.absent[e], c)));
                }
                for (int c = 0; c < C; c++) {
                    const uint64_t d = or_draw(seed, 11, b, 25u * r + e, c);
                    tern_set(&p.set[e], &p.clear[e], c,
                             mutated_state(d, m->p_rule, tern_get(p.set[e], p.clear[e], c)));
                }
            }
            if ((uint32_t)(or_draw(seed, 12, b, r, 0) >> 40) < m->p_reward) {
                const uint64_t span = (uint64_t)((int64_t)m->reward_max - m->reward_min + 1);
                p.reward = (int32_t)(m->reward_min + (int64_t)(((or_draw(seed, 12, b, r, 1) >> 32) * span) >> 32));
            }
            wr32(rec + 4, (uint32_t)p.reward);
            for (int e = 0; e < 25; e++) {
                wr32(rec + 8 + 4 * e, p.present[e]);
                wr32(rec + 108 + 4 * e, p.absent[e]);
                wr32(rec + 208 + 4 * e, p.set[e]);
                wr32(rec + 308 + 4 * e, p.clear[e]);
            }
        }
    }
    return 0;
}
