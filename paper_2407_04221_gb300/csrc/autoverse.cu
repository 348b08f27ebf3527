// autoverse.cu -- libautoverse.so: batched rewrite-rule engine for sm_103a.
//
// Host side: argument checks, rule compilation (every rule in its four
// rotations, turned into term lists over bit-planes), device buffers, launches.
// Device side: see kernels.cuh.
//
// Rule semantics follow Sec. 2.1 of Earle & Togelius, "Autoverse" (arXiv
// 2407.04221): the per-patch rule definition, the matching convolution
// ReLU(conv_{K_I}(D) - I + 1), the transposed-convolution write of the output
// pattern, force tiles for actions, and parallel application of all rules.
#include "autoverse.h"

#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <unordered_set>
#include <vector>

#include "launch.h"

using namespace av;

struct av_handle {
    DevConfig cf{};
    av_config host_cfg{};
    int n_tables = 0;
    size_t grid_bytes = 0;  // one board, canonical bytes
    // device buffers
    uint32_t *d_arena = nullptr;
    uint32_t *d_tab_off = nullptr;
    uint32_t *d_vm = nullptr;
    uint32_t *d_masks = nullptr;
    void *d_cur = nullptr;
    void *d_init = nullptr;
    int32_t *d_t = nullptr;
    uint32_t *d_cum = nullptr;
    uint32_t *d_status = nullptr;  // [0] error bits, [1] warning bits
    uint32_t *d_cost = nullptr;    // [B] memoising rollout: each environment's time in its last launch
    int32_t *d_order = nullptr;    // [B] memoising rollout: launch order (costliest environments first)
    bool order_ready = false;      // d_order holds an order (after the first memoising rollout)
    uint64_t *d_vtab = nullptr;     // [B][vis_mask + 1] visited hashes, open addressing (0 = empty)
    uint32_t *d_vzero = nullptr;    // [B] 1 if the state whose hash is 0 was visited
    int32_t *d_n_visited = nullptr; // [B]
    uint32_t vis_mask = 0;          // slots per env - 1 (a power of two >= 2 x capacity, minus one)
    uint32_t *d_rules = nullptr;    // the packed 408-byte records as given, [n_tables][R] (rule observation)
    bool large = false;             // more than AV_MAX_SMEM_CELLS cells: the band rollout
    int band_rows = 0, band_nw = 0; // rows of anchors per band, plane words per band window
    uint32_t *d_bplanes = nullptr;  // [B][C+1][NW] the boards as bit-planes during a band rollout
    uint32_t *d_bset = nullptr, *d_bclr = nullptr, *d_bbase = nullptr;  // [B][C][NW]
    VariantParams variant{};        // variant semantics (av_set_variant)
    bool variant_on = false;        // some rule is limited or inhibits another
    bool has_cum = false;
    std::string last_error;
};

namespace {

// Handles alive (created and not yet destroyed): every entry point checks its
// handle here before touching it, so a destroyed or foreign pointer gives
// AV_ESTATE instead of a use after free.
std::mutex g_handles_mu;
std::unordered_set<const av_handle *> g_handles;

bool handle_live(const av_handle *h)
{
    std::lock_guard<std::mutex> lock(g_handles_mu);
    return g_handles.count(h) != 0;
}

// AV_EINVAL for a null handle, AV_ESTATE for one that is not alive, else AV_OK.
int check_handle(const av_handle *h)
{
    if (!h)
        return AV_EINVAL;
    return handle_live(h) ? AV_OK : AV_ESTATE;
}

#define AV_HANDLE(h)                        \
    do {                                    \
        const int hc_ = check_handle(h);    \
        if (hc_ != AV_OK)                   \
            return hc_;                     \
    } while (0)

int fail(av_handle *h, int code, const std::string &msg)
{
    if (h)
        h->last_error = msg;
    return code;
}

int cuda_fail(av_handle *h, cudaError_t e, const char *where)
{
    return fail(h, AV_ECUDA, std::string(where) + ": " + cudaGetErrorString(e));
}

#define AV_CUDA(h, call)                                                                   \
    do {                                                                                   \
        cudaError_t e_ = (call);                                                           \
        if (e_ != cudaSuccess)                                                             \
            return cuda_fail((h), e_, #call);                                              \
    } while (0)

// A rule pattern as the compiler sees it (base or rotated).
struct Pat {
    int h = 0, w = 0;
    int32_t reward = 0;
    uint32_t pres[25] = {}, abs_[25] = {}, set[25] = {}, clr[25] = {};
};

Pat from_record(const av_rule &r)
{
    Pat p;
    p.h = r.h;
    p.w = r.w;
    p.reward = r.reward;
    for (int e = 0; e < 25; ++e) {
        p.pres[e] = r.present[e];
        p.abs_[e] = r.absent[e];
        p.set[e] = r.set[e];
        p.clr[e] = r.clear[e];
    }
    return p;
}

int check_config(const av_config *c, std::string &why)
{
    auto bad = [&](const char *m) { why = m; return AV_EINVAL; };
    if (c->batch < 1) return bad("batch must be >= 1");
    if (c->H < 1 || c->H > AV_MAX_SIDE || c->W < 1 || c->W > AV_MAX_SIDE) return bad("H, W must be in 1..256");
    if (c->C < 1 || c->C > AV_MAX_C) return bad("C must be in 1..16");
    if (c->n_rules < 0 || c->n_rules > AV_MAX_RULES) return bad("n_rules must be in 0..64");
    if (c->rules_per_env != 0 && c->rules_per_env != 1) return bad("rules_per_env must be 0 or 1");
    if (c->cum_per_env != 0 && c->cum_per_env != 1) return bad("cum_per_env must be 0 or 1");
    if (c->max_steps < 0) return bad("max_steps must be >= 0");
    if (c->auto_reset != 0 && c->auto_reset != 1) return bad("auto_reset must be 0 or 1");
    if (c->search_capacity < 0) return bad("search_capacity must be >= 0");
    const int32_t roles[4] = {c->ch_player, c->ch_goal, c->ch_empty, c->ch_wall};
    for (int r : roles)
        if (r < -1 || r >= c->C) return bad("role channels must be -1 or in 0..C-1");
    return AV_OK;
}

int check_rule(const av_rule &r, int C, std::string &why)
{
    if (r.h < 1 || r.h > AV_MAX_PATTERN || r.w < 1 || r.w > AV_MAX_PATTERN) {
        why = "rule h, w must be in 1..5";
        return AV_EINVAL;
    }
    const uint32_t in_ok = (C + 1 >= 32) ? 0xffffffffu : ((1u << (C + 1)) - 1u);
    const uint32_t out_ok = (1u << C) - 1u;
    for (int e = 0; e < 25; ++e) {
        const bool inside = e < r.h * r.w;
        if ((r.present[e] | r.absent[e]) & ~(inside ? in_ok : 0u)) {
            why = "rule input bits outside channels 0..C or outside the h x w pattern";
            return AV_EINVAL;
        }
        if ((r.set[e] | r.clear[e]) & ~(inside ? out_ok : 0u)) {
            why = "rule output bits outside channels 0..C-1 or outside the h x w pattern";
            return AV_EINVAL;
        }
    }
    return AV_OK;
}

// Position (i, k) of an h x w pattern after g counter-clockwise quarter turns.
void turn_position(int h, int w, int g, int &i, int &k)
{
    for (int q = 0; q < g; ++q) {
        const int ni = w - 1 - k, nk = i;
        i = ni;
        k = nk;
        const int t = h;
        h = w;
        w = t;
    }
}

// Compile one rule table into the layout read by the kernels (kernels.cuh,
// "Rule table layout").  The term order is chosen once on the base pattern
// and carried through every rotation, so the four rotations of a rule run
// the same loop.  Any order gives the same result; a selective order lets
// evaluation stop early.  Present terms: an exclusive pair of present tile
// channels first (see below), then a present force term, positions with more
// present channels, the player channel, then rarer channels.  Absent terms
// follow: first those at positions with no present tile channel (at a
// position whose tile is already fixed by a present term, an absent tile
// channel almost always holds), the most common channels first.  `density`
// (C entries, or null) is each tile channel's share of cells in the initial
// maps; without it every tile channel counts as equally common.
void compile_table(const av_rule *rules, const DevConfig &cf, const double *density, std::vector<uint32_t> &arena,
                   double *live_rules)
{
    *live_rules = 0.0;
    const size_t base = arena.size();
    const int R = cf.R;
    std::vector<uint32_t> hdr(8 * (size_t)R, 0), terms, outs;
    uint32_t n_terms = 0, n_outs = 0;
    // how common a channel is on a cell: the force and the player mark one cell
    auto common = [&](int c) -> double {
        if (c == cf.C || c == cf.ch_player)
            return 1.0 / cf.HW;
        return density ? density[c] : 1.0 / cf.C;
    };
    for (int r = 0; r < R; ++r) {
        const Pat p = from_record(rules[r]);
        struct BT { int i, k, c, neg, key0, key1; double dens; };
        std::vector<BT> pres, absn;
        for (int i = 0; i < p.h; ++i)
            for (int k = 0; k < p.w; ++k) {
                const int e = i * p.w + k;
                const int npos = __builtin_popcount(p.pres[e]);
                uint32_t tiles = p.pres[e] & ((1u << cf.C) - 1u);
                if (cf.ch_player >= 0)
                    tiles &= ~(1u << cf.ch_player);
                for (int c = 0; c <= cf.C; ++c) {
                    const int rank = c == cf.C ? 2 : (c == cf.ch_player ? 1 : 0);
                    const int key0 = c == cf.C ? 100 + npos : npos;  // a present force term first
                    if ((p.pres[e] >> c) & 1u) pres.push_back({i, k, c, 0, key0, rank, common(c)});
                    if ((p.abs_[e] >> c) & 1u) absn.push_back({i, k, c, 1, tiles ? 1 : 0, 0, common(c)});
                }
            }
        std::stable_sort(pres.begin(), pres.end(), [](const BT &a, const BT &b) {
            if (a.key0 != b.key0) return a.key0 > b.key0;
            if (a.key0 > 1 && a.key0 < 100 && a.i * 8 + a.k != b.i * 8 + b.k)
                return a.i * 8 + a.k < b.i * 8 + b.k;  // keep a position's present terms together
            if (a.key1 != b.key1) return a.key1 > b.key1;
            if (a.dens != b.dens) return a.dens < b.dens;
            return a.c > b.c;
        });
        std::stable_sort(absn.begin(), absn.end(), [](const BT &a, const BT &b) {
            if (a.key0 != b.key0) return a.key0 < b.key0;  // positions without a present tile first
            return a.dens > b.dens;
        });
        // An exclusive pair leads when the rule has one: two present tile
        // channels (neither the player's) at one position.  Initial maps hold
        // one tile type per cell (the player overlays), so such a pair rules
        // out every anchor at once until rules make cells multi-hot.
        for (int i = 0, found = 0; i < p.h && !found; ++i)
            for (int k = 0; k < p.w && !found; ++k) {
                int picks[2], n = 0;
                for (size_t u = 0; u < pres.size() && n < 2; ++u)
                    if (pres[u].i == i && pres[u].k == k && pres[u].c < cf.C && pres[u].c != cf.ch_player)
                        picks[n++] = (int)u;
                if (n == 2) {
                    const BT a = pres[picks[0]], b = pres[picks[1]];
                    pres.erase(pres.begin() + picks[1]);
                    pres.erase(pres.begin() + picks[0]);
                    pres.insert(pres.begin(), b);
                    pres.insert(pres.begin(), a);
                    found = 1;
                }
            }
        // Expected anchors per step that pass the rule's first kRegTerms
        // present terms, channels taken as independent with the densities above
        // (an exclusive pair passes nowhere), capped at one: the expected chance
        // that the rule needs more than its register-resident terms in a step.
        {
            double pass = 1.0;
            const size_t nreg = std::min(pres.size(), (size_t)kRegTerms);
            const bool exclusive = nreg >= 2 && pres[0].i == pres[1].i && pres[0].k == pres[1].k &&
                                   pres[0].c < cf.C && pres[1].c < cf.C && pres[0].c != cf.ch_player &&
                                   pres[1].c != cf.ch_player;
            for (size_t j = 0; j < nreg; ++j)
                pass *= pres[j].dens;
            if (exclusive)
                pass = 0.0;
            double anchors = 0.0;
            for (int g = 0; g < 4; ++g) {
                const int hh = (g & 1) ? p.w : p.h, ww = (g & 1) ? p.h : p.w;
                anchors += (double)std::max(0, cf.H - hh + 1) * std::max(0, cf.W - ww + 1);
            }
            *live_rules += std::min(1.0, anchors * pass);
        }
        uint32_t *hd = &hdr[8 * (size_t)r];
        hd[0] = (uint32_t)pres.size();
        hd[1] = (uint32_t)absn.size();
        hd[3] = (uint32_t)p.reward;
        hd[4] = n_terms;
        hd[5] = n_outs;
        uint32_t shapes = 0;
        for (int g = 0; g < 4; ++g) {
            const int hh = (g & 1) ? p.w : p.h, ww = (g & 1) ? p.h : p.w;
            shapes |= (uint32_t)((hh - 1) * AV_MAX_PATTERN + (ww - 1)) << (8 * g);
        }
        hd[6] = shapes;
        std::vector<BT> all(pres);
        all.insert(all.end(), absn.begin(), absn.end());
        for (const BT &t : all) {
            for (int g = 0; g < 4; ++g) {
                int i = t.i, k = t.k;
                turn_position(p.h, p.w, g, i, k);
                const int s = i * cf.W + k;
                terms.push_back((uint32_t)((t.c * cf.NWP + (s >> 5)) * 8));
                terms.push_back((uint32_t)(s & 31) | (t.neg ? kTermAbsent : 0u));
            }
            ++n_terms;
        }
        // padding: the terms after the first kRegTerms present ones fill whole batches
        const int after = (int)all.size() - std::min((int)pres.size(), kRegTerms);
        for (int j = after; j % kRestBatch != 0; ++j) {
            for (int g = 0; g < 4; ++g) {
                terms.push_back((uint32_t)((cf.C + 1) * cf.NWP * 8));
                terms.push_back(kTermAbsent);
            }
            ++n_terms;
        }
        uint32_t no = 0;
        for (int i0 = 0; i0 < p.h; ++i0)
            for (int k0 = 0; k0 < p.w; ++k0) {
                const int e = i0 * p.w + k0;
                if (!(p.set[e] | p.clr[e]))
                    continue;
                for (int g = 0; g < 4; ++g) {
                    int i = i0, k = k0;
                    turn_position(p.h, p.w, g, i, k);
                    const int s = i * cf.W + k;
                    outs.push_back((uint32_t)(s >> 5));
                    outs.push_back((uint32_t)(s & 31));
                    outs.push_back(p.set[e]);
                    outs.push_back(p.clr[e]);
                }
                ++no;
            }
        hd[2] = no;
        n_outs += no;
    }
    // one batch of passing terms after the last rule's: a read one batch past
    // any rule's terms stays inside the term list
    for (int j = 0; j < kRestBatch; ++j) {
        for (int g = 0; g < 4; ++g) {
            terms.push_back((uint32_t)((cf.C + 1) * cf.NWP * 8));
            terms.push_back(kTermAbsent);
        }
        ++n_terms;
    }
    const uint32_t tw = table_terms_word(R), ow = table_outs_word(R, n_terms);
    arena.resize(base + ow + outs.size(), 0);
    uint32_t *t = &arena[base];
    t[0] = (uint32_t)R;
    t[1] = n_terms;
    t[2] = n_outs;
    std::copy(hdr.begin(), hdr.end(), t + 4);
    std::copy(terms.begin(), terms.end(), t + tw);
    std::copy(outs.begin(), outs.end(), t + ow);
    while (arena.size() & 3u) arena.push_back(0);  // next table starts 16-byte aligned
}

// Column and cell masks over plane words: first column, last column, cells < H*W.
std::vector<uint32_t> column_masks(const DevConfig &cf)
{
    std::vector<uint32_t> m(3 * (size_t)cf.NW, 0);
    for (int p = 0; p < cf.HW; ++p) {
        const int x = p % cf.W, w = p >> 5;
        const uint32_t bit = 1u << (p & 31);
        if (x == 0) m[w] |= bit;
        if (x == cf.W - 1) m[cf.NW + w] |= bit;
        m[2 * cf.NW + w] |= bit;
    }
    return m;
}

// Valid-anchor masks: vm[shape][word] bit b set when anchor p = 32*word + b
// has its h' x w' window inside the board.
std::vector<uint32_t> valid_masks(const DevConfig &cf)
{
    std::vector<uint32_t> vm((size_t)kShapes * cf.NW, 0);
    for (int hh = 1; hh <= AV_MAX_PATTERN; ++hh)
        for (int ww = 1; ww <= AV_MAX_PATTERN; ++ww) {
            const int shape = (hh - 1) * AV_MAX_PATTERN + (ww - 1);
            for (int p = 0; p < cf.HW; ++p) {
                const int y = p / cf.W, x = p % cf.W;
                if (y <= cf.H - hh && x <= cf.W - ww)
                    vm[(size_t)shape * cf.NW + (p >> 5)] |= 1u << (p & 31);
            }
        }
    return vm;
}

template <typename T>
int dalloc(av_handle *h, T **p, size_t n)
{
    if (getenv("AV_FAIL_ALLOC"))  // host-side fault injection for the ENOMEM path
        return fail(h, AV_ENOMEM, "allocation refused (AV_FAIL_ALLOC set)");
    cudaError_t e = cudaMalloc((void **)p, n * sizeof(T) + (n == 0 ? 8 : 0));
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(h, e == cudaErrorMemoryAllocation ? AV_ENOMEM : AV_ECUDA,
                    std::string("cudaMalloc: ") + cudaGetErrorString(e));
    }
    return AV_OK;
}

void free_all(av_handle *h)
{
    cudaFree(h->d_arena);
    cudaFree(h->d_tab_off);
    cudaFree(h->d_vm);
    cudaFree(h->d_masks);
    cudaFree(h->d_cur);
    cudaFree(h->d_init);
    cudaFree(h->d_t);
    cudaFree(h->d_cum);
    cudaFree(h->d_status);
    cudaFree(h->d_cost);
    cudaFree(h->d_order);
    cudaFree(h->d_vtab);
    cudaFree(h->d_vzero);
    cudaFree(h->d_n_visited);
    cudaFree(h->d_rules);
    cudaFree(h->d_bplanes);
    cudaFree(h->d_bset);
    cudaFree(h->d_bclr);
    cudaFree(h->d_bbase);
}

cudaStream_t as_stream(uintptr_t s) { return reinterpret_cast<cudaStream_t>(s); }

int launch_check(av_handle *h, const char *what)
{
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return cuda_fail(h, e, what);
    return AV_OK;
}

}  // namespace

// ---------------------------------------------------------------- C ABI
extern "C" {

const char *av_strerror(int s)
{
    switch (s) {
    case AV_OK: return "ok";
    case AV_EINVAL: return "invalid argument";
    case AV_ENOMEM: return "out of memory";
    case AV_ECUDA: return "CUDA error";
    case AV_ESTATE: return "invalid handle state";
    case AV_EDEVICE: return "device-side error";
    default: return "unknown status";
    }
}

const char *av_last_error(av_handle *h)
{
    if (!h)
        return "null handle";
    return handle_live(h) ? h->last_error.c_str() : "not a live handle (destroyed or never created)";
}

int av_create(const av_config *cfg, const av_rule *rules, av_handle **out)
{
    if (!cfg || !out || (cfg->n_rules > 0 && !rules))
        return AV_EINVAL;
    *out = nullptr;
    std::string why;
    if (check_config(cfg, why) != AV_OK)
        return AV_EINVAL;
    const int n_tables = cfg->rules_per_env ? cfg->batch : 1;
    for (size_t i = 0; i < (size_t)n_tables * cfg->n_rules; ++i)
        if (check_rule(rules[i], cfg->C, why) != AV_OK)
            return AV_EINVAL;

    av_handle *h = new (std::nothrow) av_handle();
    if (!h)
        return AV_ENOMEM;
    h->host_cfg = *cfg;
    h->host_cfg.init_cum = nullptr;
    h->n_tables = n_tables;
    DevConfig &cf = h->cf;
    cf.B = cfg->batch;
    cf.H = cfg->H;
    cf.W = cfg->W;
    cf.C = cfg->C;
    cf.HW = cfg->H * cfg->W;
    cf.NW = (cf.HW + 31) / 32;
    cf.NA = anchor_slots(cf.NW);
    cf.NWP = 8 * cf.NA + kPlanePad;
    if (cf.HW > AV_MAX_SMEM_CELLS) {
        // bands of rows through shared memory: the rule tables address the
        // band window's planes, the lanes cover its words
        h->large = true;
        band_geometry(cf.H, cf.W, &h->band_rows, &h->band_nw, &cf.NA, &cf.NWP);
    }
    cf.R = cfg->n_rules;
    cf.rules_per_env = cfg->rules_per_env;
    cf.max_steps = cfg->max_steps;
    cf.auto_reset = cfg->auto_reset;
    cf.ch_player = cfg->ch_player;
    cf.ch_goal = cfg->ch_goal;
    cf.ch_empty = cfg->ch_empty;
    cf.ch_wall = cfg->ch_wall;
    cf.border_wall = cfg->border_wall ? 1 : 0;
    cf.cum_per_env = cfg->cum_per_env;
    cf.cell_bytes = cfg->C <= 8 ? 1 : 2;
    // Kernel path override, for testing every path on the same shapes:
    // AV_KERNEL_PATH selects a rollout kernel for tests and measurements:
    // block (one CTA per env), fast (several warps per env) or warp (one warp
    // per env); by default the library chooses.  AV_FAST_WARPS=8 runs the fast
    // rollout with 8 warps per env.
    if (const char *path = getenv("AV_KERNEL_PATH"))
        cf.path = strcmp(path, "block") == 0  ? 1
                  : strcmp(path, "fast") == 0 ? 2
                  : strcmp(path, "warp") == 0 ? 3
                  : strcmp(path, "memo") == 0 ? 4
                                              : 0;
    // AV_MEMO_STAGE=1 or 0: the memoising rollout copies the rule tables into
    // shared memory, or reads them through the L1 cache (default: decided by size).
    if (const char *ms = getenv("AV_MEMO_STAGE"))
        cf.memo_stage = atoi(ms) ? 1 : 2;
    // AV_MEMO_WARPS=1|2|4|8: warps per environment of the memoising rollout.
    if (const char *mw = getenv("AV_MEMO_WARPS"))
        cf.memo_warps = atoi(mw);
    if (const char *fw = getenv("AV_FAST_WARPS"))
        cf.fast_warps = atoi(fw) == 8 ? 8 : 4;
    h->grid_bytes = (size_t)cf.HW * cf.cell_bytes;

    std::vector<uint32_t> arena, tab_off((size_t)n_tables + 1);
    uint32_t max_words = 0;
    double live_sum = 0.0;  // expected rules per step that pass their register terms, summed over tables
    // tile-channel densities of the initial maps, per table, for the term order
    std::vector<double> density;
    if (cfg->init_cum) {
        const int n_cum = cfg->cum_per_env ? cf.B : 1;
        density.assign((size_t)n_cum * cf.C, 0.0);
        for (int e = 0; e < n_cum; ++e)
            for (int c = 0; c < cf.C; ++c) {
                const uint32_t hi = cfg->init_cum[(size_t)e * cf.C + c];
                const uint32_t lo = c ? cfg->init_cum[(size_t)e * cf.C + c - 1] : 0u;
                density[(size_t)e * cf.C + c] = hi > lo ? (double)(hi - lo) / 16777216.0 : 0.0;
            }
        if (n_cum > 1 && n_tables == 1) {  // one shared table: the mean over environments
            for (int e = 1; e < n_cum; ++e)
                for (int c = 0; c < cf.C; ++c)
                    density[c] += density[(size_t)e * cf.C + c];
            density.resize(cf.C);
            for (double &d : density)
                d /= n_cum;
        }
    }
    for (int t = 0; t < n_tables; ++t) {
        tab_off[t] = (uint32_t)arena.size();
        const double *dens = nullptr;
        if (!density.empty())
            dens = density.data() + (density.size() > (size_t)cf.C && n_tables == cf.B ? (size_t)t * cf.C : 0);
        double live = 0.0;
        compile_table(rules + (size_t)t * cfg->n_rules, cf, dens, arena, &live);
        live_sum += live;
        max_words = std::max(max_words, (uint32_t)arena.size() - tab_off[t]);
    }
    tab_off[n_tables] = (uint32_t)arena.size();
    // Environments whose rules keep passing their register-resident terms step
    // after step do most of their work in the one-warp kernel's general step,
    // one rule after another; the block kernel spreads the rules over eight
    // warps.  Busy when, on average, an environment expects half a rule or
    // more per step to get past its register terms.
    cf.busy = live_sum / n_tables >= 0.5 ? 1 : 0;
    cf.rule_words = max_words <= (uint32_t)kMaxSmemRuleWords ? (int)max_words : 0;
    std::vector<uint32_t> vm = valid_masks(cf);
    std::vector<uint32_t> masks = column_masks(cf);

    int rc;
    const size_t B = (size_t)cf.B;
    if ((rc = dalloc(h, &h->d_arena, arena.size())) || (rc = dalloc(h, &h->d_tab_off, tab_off.size())) ||
        (rc = dalloc(h, &h->d_vm, vm.size())) || (rc = dalloc(h, &h->d_masks, masks.size())) ||
        (rc = dalloc(h, (uint8_t **)&h->d_cur, B * h->grid_bytes)) ||
        (rc = dalloc(h, (uint8_t **)&h->d_init, B * h->grid_bytes)) || (rc = dalloc(h, &h->d_t, B)) ||
        (rc = dalloc(h, &h->d_status, 4)) || (rc = dalloc(h, &h->d_cost, B)) || (rc = dalloc(h, &h->d_order, B)) ||
        (rc = dalloc(h, (uint8_t **)&h->d_rules, (size_t)n_tables * cfg->n_rules * sizeof(av_rule)))) {
        free_all(h);
        delete h;
        return rc;
    }
    if (cfg->init_cum) {
        const size_t ncum = (size_t)(cfg->cum_per_env ? cf.B : 1) * cf.C;
        if ((rc = dalloc(h, &h->d_cum, ncum)) ||
            cudaMemcpy(h->d_cum, cfg->init_cum, ncum * 4, cudaMemcpyHostToDevice) != cudaSuccess) {
            free_all(h);
            delete h;
            return rc ? rc : AV_ECUDA;
        }
        h->has_cum = true;
    }
    if (h->large) {
        const size_t words = B * (size_t)cf.NW;
        if ((rc = dalloc(h, &h->d_bplanes, words * (cf.C + 1))) || (rc = dalloc(h, &h->d_bset, words * cf.C)) ||
            (rc = dalloc(h, &h->d_bclr, words * cf.C)) || (rc = dalloc(h, &h->d_bbase, words * cf.C))) {
            free_all(h);
            delete h;
            return rc;
        }
    }
    if (cfg->search_capacity > 0) {
        size_t slots = 64;
        while (slots < 2 * (size_t)cfg->search_capacity)
            slots <<= 1;
        h->vis_mask = (uint32_t)(slots - 1);
        if ((rc = dalloc(h, &h->d_vtab, B * slots)) || (rc = dalloc(h, &h->d_vzero, B)) ||
            (rc = dalloc(h, &h->d_n_visited, B))) {
            free_all(h);
            delete h;
            return rc;
        }
        cudaMemset(h->d_n_visited, 0, B * 4);
    }
    cudaError_t e = cudaSuccess;
    if (e == cudaSuccess) e = cudaMemcpy(h->d_arena, arena.data(), arena.size() * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(h->d_tab_off, tab_off.data(), tab_off.size() * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(h->d_vm, vm.data(), vm.size() * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(h->d_masks, masks.data(), masks.size() * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess && cfg->n_rules > 0)
        e = cudaMemcpy(h->d_rules, rules, (size_t)n_tables * cfg->n_rules * sizeof(av_rule), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemset(h->d_cur, 0, B * h->grid_bytes);
    if (e == cudaSuccess) e = cudaMemset(h->d_init, 0, B * h->grid_bytes);
    if (e == cudaSuccess) e = cudaMemset(h->d_t, 0, B * 4);
    if (e == cudaSuccess) e = cudaMemset(h->d_status, 0, 16);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        free_all(h);
        delete h;
        return AV_ECUDA;
    }
    if (configure_kernels() != cudaSuccess) {
        free_all(h);
        delete h;
        return AV_ECUDA;
    }
    {
        std::lock_guard<std::mutex> lock(g_handles_mu);
        g_handles.insert(h);
    }
    *out = h;
    return AV_OK;
}

int av_destroy(av_handle *h)
{
    if (!h)
        return AV_EINVAL;
    {
        std::lock_guard<std::mutex> lock(g_handles_mu);
        if (!g_handles.erase(h))
            return AV_ESTATE;  // destroyed already, or never created
    }
    cudaDeviceSynchronize();
    free_all(h);
    delete h;
    return AV_OK;
}

int av_reset(av_handle *h, uint64_t seed, void *obs, uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h)
        return AV_EINVAL;
    if (!h->has_cum)
        return fail(h, AV_ESTATE, "av_reset: the handle was created without init_cum");
    launch_reset(h->cf, h->d_cum, seed, h->d_cur, h->d_init, h->d_t, obs, as_stream(stream));
    return launch_check(h, "reset kernel");
}

int av_set_state(av_handle *h, const void *grids, const int32_t *t, int set_as_init, uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h || !grids)
        return AV_EINVAL;
    cudaStream_t s = as_stream(stream);
    const size_t n = (size_t)h->cf.B * h->grid_bytes;
    AV_CUDA(h, cudaMemcpyAsync(h->d_cur, grids, n, cudaMemcpyDeviceToDevice, s));
    if (set_as_init)
        AV_CUDA(h, cudaMemcpyAsync(h->d_init, grids, n, cudaMemcpyDeviceToDevice, s));
    if (t)
        AV_CUDA(h, cudaMemcpyAsync(h->d_t, t, (size_t)h->cf.B * 4, cudaMemcpyDeviceToDevice, s));
    else
        AV_CUDA(h, cudaMemsetAsync(h->d_t, 0, (size_t)h->cf.B * 4, s));
    return AV_OK;
}

int av_get_state(av_handle *h, void *grids, int32_t *t, uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h || !grids)
        return AV_EINVAL;
    cudaStream_t s = as_stream(stream);
    AV_CUDA(h, cudaMemcpyAsync(grids, h->d_cur, (size_t)h->cf.B * h->grid_bytes,
                               cudaMemcpyDeviceToDevice, s));
    if (t)
        AV_CUDA(h, cudaMemcpyAsync(t, h->d_t, (size_t)h->cf.B * 4, cudaMemcpyDeviceToDevice, s));
    return AV_OK;
}

int av_step(av_handle *h, const uint8_t *actions, void *obs, int32_t *reward, uint8_t *done,
            uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h || !actions)
        return AV_EINVAL;
    if (h->large) {
        launch_rollout_band(h->cf, h->band_rows, h->band_nw, h->d_arena, h->d_tab_off, h->d_vm, h->d_masks,
                            h->d_cur, h->d_init, h->d_t, 1, 0, actions, obs, reward, done, nullptr, h->d_status,
                            h->d_bplanes, h->d_bset, h->d_bclr, h->d_bbase, as_stream(stream));
        return launch_check(h, "band step kernel");
    }
    if (h->variant_on) {
        launch_rollout_variant(h->cf, h->variant, h->d_arena, h->d_tab_off, h->d_vm, h->d_masks, h->d_cur,
                               h->d_init, h->d_t, 1, 0, actions, obs, reward, done, nullptr, h->d_status,
                               as_stream(stream));
        return launch_check(h, "variant step kernel");
    }
    launch_rollout(h->cf, h->d_arena, h->d_tab_off, h->d_vm, h->d_masks, h->d_cur, h->d_init, h->d_t, 1, 0,
                   actions, obs, reward, done, nullptr, h->d_status, as_stream(stream));
    return launch_check(h, "step kernel");
}

int av_rollout(av_handle *h, int32_t n_steps, uint64_t action_seed, void *obs_traj,
               int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h || n_steps < 0)
        return AV_EINVAL;
    if (n_steps == 0)
        return AV_OK;
    if (h->large) {
        launch_rollout_band(h->cf, h->band_rows, h->band_nw, h->d_arena, h->d_tab_off, h->d_vm, h->d_masks,
                            h->d_cur, h->d_init, h->d_t, n_steps, action_seed, nullptr, obs_traj, rew_traj,
                            done_traj, rew_sum, h->d_status, h->d_bplanes, h->d_bset, h->d_bclr, h->d_bbase,
                            as_stream(stream));
        return launch_check(h, "band rollout kernel");
    }
    if (h->variant_on) {
        launch_rollout_variant(h->cf, h->variant, h->d_arena, h->d_tab_off, h->d_vm, h->d_masks, h->d_cur,
                               h->d_init, h->d_t, n_steps, action_seed, nullptr, obs_traj, rew_traj, done_traj,
                               rew_sum, h->d_status, as_stream(stream));
        return launch_check(h, "variant rollout kernel");
    }
    // The memoising rollout takes the environments that cost most in its last
    // launch first (their cost comes mostly from their rules, so it carries
    // over); the order changes no result, environments being independent.
    const bool memo = use_memo_rollout(h->cf);
    launch_rollout(h->cf, h->d_arena, h->d_tab_off, h->d_vm, h->d_masks, h->d_cur, h->d_init, h->d_t, n_steps,
                   action_seed, nullptr, obs_traj, rew_traj, done_traj, rew_sum, h->d_status,
                   as_stream(stream), memo && h->order_ready ? h->d_order : nullptr, memo ? h->d_cost : nullptr);
    int rc = launch_check(h, "rollout kernel");
    if (rc == AV_OK && memo) {
        launch_memo_order(h->d_cost, h->d_order, h->cf.B, as_stream(stream));
        rc = launch_check(h, "launch order kernel");
        h->order_ready = rc == AV_OK;
    }
    return rc;
}

int av_expand(av_handle *h, const void *parents, int32_t F, const int32_t *n_parent,
              void *children, int32_t *rewards, uint8_t *done, uint64_t *hashes,
              uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h || F < 0 || (F > 0 && (!parents || !children || !rewards || !hashes)))
        return AV_EINVAL;
    if ((size_t)h->cf.B * (size_t)F > 0x7fffffffu)
        return AV_EINVAL;
    if (h->large)
        return fail(h, AV_EINVAL, "av_expand: boards over AV_MAX_SMEM_CELLS cells are not supported");
    if (F == 0)
        return AV_OK;
    if (h->variant_on)
        return fail(h, AV_ESTATE, "av_expand: variant semantics are set (av_set_variant); expansion uses the standard step");
    launch_expand(h->cf, h->d_arena, h->d_tab_off, h->d_vm, h->d_masks, parents, F, n_parent, children, rewards,
                  done, hashes, as_stream(stream));
    return launch_check(h, "expand kernel");
}

int av_observe(av_handle *h, const void *grids, int32_t window, uint8_t *obs, int32_t *player_yx,
               uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h || !obs)
        return AV_EINVAL;
    if (window < 1 || window > AV_MAX_WINDOW)
        return fail(h, AV_EINVAL, "av_observe: window must be in 1..AV_MAX_WINDOW");
    if (h->cf.ch_player < 0)
        return fail(h, AV_ESTATE, "av_observe: the configuration has no player channel");
    if ((size_t)h->cf.B > 0x7fffffffu)
        return AV_EINVAL;
    launch_observe(h->cf, grids ? grids : h->d_cur, window, obs, player_yx, as_stream(stream));
    return launch_check(h, "observe kernel");
}

int av_rule_obs(av_handle *h, uint8_t *bits, int32_t *reward, uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h || (!bits && h->cf.R > 0))
        return AV_EINVAL;
    const size_t n = (size_t)h->n_tables * h->cf.R;
    if (n * 100 > 0x7fffffffu)
        return AV_EINVAL;
    launch_rule_obs((int)n, h->cf.C, h->d_rules, bits, reward, as_stream(stream));
    return launch_check(h, "rule observation kernel");
}

int av_set_variant(av_handle *h, const av_variant *v)
{
    AV_HANDLE(h);
    if (!h)
        return AV_EINVAL;
    VariantParams p{};
    bool on = false;
    if (v) {
        const int R = h->cf.R;
        const uint64_t rules = R >= 64 ? ~0ull : ((1ull << R) - 1ull);
        if (v->random_keys != 0 && v->random_keys != 1)
            return fail(h, AV_EINVAL, "av_set_variant: random_keys must be 0 or 1");
        for (int r = 0; r < AV_MAX_RULES; ++r) {
            if (v->limit[r] < 0 || v->limit[r] > AV_MAX_LIMIT)
                return fail(h, AV_EINVAL, "av_set_variant: limits must be in 0..AV_MAX_LIMIT");
            if (r >= R && (v->limit[r] != 0 || v->inhibit[r] != 0))
                return fail(h, AV_EINVAL, "av_set_variant: limit or inhibit set for a rule slot >= n_rules");
            if (v->inhibit[r] & ~rules)
                return fail(h, AV_EINVAL, "av_set_variant: inhibit mask names a rule slot >= n_rules");
            p.limit[r] = v->limit[r];
            p.inhibit[r] = v->inhibit[r];
            on = on || v->limit[r] != 0 || v->inhibit[r] != 0;
        }
        p.random_keys = v->random_keys;
        p.key_seed = v->key_seed;
        if (on && h->large)
            return fail(h, AV_EINVAL, "av_set_variant: boards over AV_MAX_SMEM_CELLS cells are not supported");
    }
    h->variant = p;
    h->variant_on = on;
    return AV_OK;
}

int av_mutate(int32_t batch, int32_t H, int32_t W, int32_t C, int32_t n_rules, const av_mutation *m,
              uint64_t seed, void *maps, av_rule *rules, uintptr_t stream)
{
    if (!m || batch < 1 || H < 1 || H > AV_MAX_SIDE || W < 1 || W > AV_MAX_SIDE || C < 1 || C > AV_MAX_C ||
        n_rules < 0 || n_rules > AV_MAX_RULES)
        return AV_EINVAL;
    const uint32_t one = 1u << 24;
    if (m->p_map > one || m->p_rule > one || m->p_reward > one || m->reward_min > m->reward_max)
        return AV_EINVAL;
    launch_mutate(batch, H, W, C, n_rules, m->p_map, m->map_channels, m->p_rule, m->p_reward, m->reward_min,
                  m->reward_max, m->mutable_rules, seed, maps, reinterpret_cast<uint32_t *>(rules),
                  as_stream(stream));
    const cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? AV_OK : AV_ECUDA;
}

int av_search_init(av_handle *h, const void *roots, uint64_t *root_hash, uint8_t *root_live,
                   uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h || !roots || !root_hash || !root_live)
        return AV_EINVAL;
    if (h->host_cfg.search_capacity < 1)
        return fail(h, AV_ESTATE, "av_search_init: search_capacity is 0");
    if (h->large)
        return fail(h, AV_EINVAL, "av_search_init: boards over AV_MAX_SMEM_CELLS cells are not supported");
    const cudaStream_t st = as_stream(stream);
    AV_CUDA(h, cudaMemsetAsync(h->d_vtab, 0, (size_t)h->cf.B * (h->vis_mask + 1) * sizeof(uint64_t), st));
    AV_CUDA(h, cudaMemsetAsync(h->d_vzero, 0, (size_t)h->cf.B * sizeof(uint32_t), st));
    launch_search_init(h->cf, h->vis_mask, roots, root_hash, root_live, h->d_vtab, h->d_vzero, h->d_n_visited,
                       st);
    return launch_check(h, "search init kernel");
}

int av_select(av_handle *h, int32_t F, const int32_t *n_parent, const int32_t *parent_cum,
              const uint8_t *parent_live, const void *cand_grids, const int32_t *cand_reward,
              const uint8_t *cand_done, const uint64_t *cand_hash, int32_t k, void *next_grids,
              int32_t *next_cum, uint64_t *next_hash, uint8_t *next_live, int32_t *n_next,
              uintptr_t stream)
{
    AV_HANDLE(h);
    if (!h)
        return AV_EINVAL;
    if (h->host_cfg.search_capacity < 1)
        return fail(h, AV_ESTATE, "av_select: search_capacity is 0");
    if (h->large)
        return fail(h, AV_EINVAL, "av_select: boards over AV_MAX_SMEM_CELLS cells are not supported");
    if (F < 1 || 5 * F > kMaxCand || k < 1 || k > 5 * F)
        return fail(h, AV_EINVAL, "av_select: need 1 <= F, 5*F <= 4096, 1 <= k <= 5*F");
    if (!n_parent || !parent_cum || !parent_live || !cand_grids || !cand_reward || !cand_done ||
        !cand_hash || !next_grids || !next_cum || !next_hash || !next_live || !n_next)
        return AV_EINVAL;
    launch_select_hash(h->cf, h->host_cfg.search_capacity, h->vis_mask, F, n_parent, parent_cum, parent_live,
                       cand_grids, cand_reward, cand_done, cand_hash, k, next_grids, next_cum, next_hash,
                       next_live, n_next, h->d_vtab, h->d_vzero, h->d_n_visited, h->d_status,
                       as_stream(stream));
    return launch_check(h, "select kernel");
}

}  // extern "C"

// ------------------------------------------------ av_select without allocation
namespace {

// Working copy of the visited sets for av_select_static: [2][batch][capacity]
// (input copy, merged result) followed by a status word.  Lives as long as the
// process, on every GPU that loads the library.
constexpr size_t kStaticHashes = AV_SELECT_STATIC_MAX_HASHES;
__device__ __align__(256) uint64_t g_select_scratch[kStaticHashes + 32];

constexpr int kMaxDevices = 64;
uint64_t *g_scratch_ptr[kMaxDevices] = {};  // device address of g_select_scratch, per device
bool g_scratch_ready[kMaxDevices] = {};

// Once per device, with it current: look up the array's device address (in
// host code the symbol is only a stand-in) and allow select's shared memory.
int static_scratch(uint64_t **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return AV_ECUDA;
    if (!g_scratch_ready[dev]) {
        void *ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_select_scratch) != cudaSuccess || !ptr)
            return AV_ECUDA;
        if (configure_search() != cudaSuccess)
            return AV_ECUDA;
        g_scratch_ptr[dev] = static_cast<uint64_t *>(ptr);
        g_scratch_ready[dev] = true;
    }
    *out = g_scratch_ptr[dev];
    return AV_OK;
}

}  // namespace

extern "C" {

int av_select_static(int32_t batch, int32_t H, int32_t W, int32_t C, int32_t F,
                     const int32_t *n_parent, const int32_t *parent_cum,
                     const uint8_t *parent_live, const void *cand_grids,
                     const int32_t *cand_reward, const uint8_t *cand_done,
                     const uint64_t *cand_hash, int32_t k, void *next_grids, int32_t *next_cum,
                     uint64_t *next_hash, uint8_t *next_live, int32_t *n_next, uint64_t *visited,
                     int32_t *n_visited, int32_t capacity, uint32_t *status, uintptr_t stream)
{
    if (batch < 1 || H < 1 || H > AV_MAX_SIDE || W < 1 || W > AV_MAX_SIDE || C < 1 || C > AV_MAX_C ||
        H * W > AV_MAX_SMEM_CELLS)
        return AV_EINVAL;
    if (F < 1 || 5 * F > kMaxCand || k < 1 || k > 5 * F || capacity < 1)
        return AV_EINVAL;
    if (2 * (size_t)batch * (size_t)capacity > kStaticHashes)
        return AV_EINVAL;  // beyond the fixed working array
    if (!n_parent || !parent_cum || !parent_live || !cand_grids || !cand_reward || !cand_done ||
        !cand_hash || !next_grids || !next_cum || !next_hash || !next_live || !n_next || !visited ||
        !n_visited)
        return AV_EINVAL;
    uint64_t *scratch = nullptr;
    int rc = static_scratch(&scratch);
    if (rc != AV_OK)
        return rc;
    DevConfig cf{};
    cf.B = batch;
    cf.H = H;
    cf.W = W;
    cf.C = C;
    cf.HW = H * W;
    cf.cell_bytes = C <= 8 ? 1 : 2;
    cudaStream_t st = as_stream(stream);
    const size_t n = (size_t)batch * capacity;
    uint32_t *sstatus = reinterpret_cast<uint32_t *>(scratch + kStaticHashes);
    if (cudaMemsetAsync(sstatus, 0, 4, st) != cudaSuccess ||
        cudaMemcpyAsync(scratch, visited, n * 8, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return AV_ECUDA;
    launch_select(cf, capacity, 0, F, n_parent, parent_cum, parent_live, cand_grids, cand_reward,
                  cand_done, cand_hash, k, next_grids, next_cum, next_hash, next_live, n_next, scratch,
                  n_visited, sstatus, st);
    if (cudaGetLastError() != cudaSuccess)
        return AV_ECUDA;
    if (cudaMemcpyAsync(visited, scratch + n, n * 8, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return AV_ECUDA;
    if (status && cudaMemcpyAsync(status, sstatus, 4, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return AV_ECUDA;
    return AV_OK;
}

int av_sync(av_handle *h)
{
    AV_HANDLE(h);
    if (!h)
        return AV_EINVAL;
    AV_CUDA(h, cudaDeviceSynchronize());
    uint32_t st[2] = {0, 0};
    AV_CUDA(h, cudaMemcpy(st, h->d_status, 8, cudaMemcpyDeviceToHost));
    if (st[0]) {
        char buf[96];
        snprintf(buf, sizeof buf, "device status 0x%x (bit 0: visited-set overflow)", st[0]);
        AV_CUDA(h, cudaMemset(h->d_status, 0, 4));
        return fail(h, AV_EDEVICE, buf);
    }
    return AV_OK;
}

int av_rollout_path(av_handle *h, int32_t *path)
{
    AV_HANDLE(h);
    if (!h || !path)
        return AV_EINVAL;
    *path = h->large                   ? AV_PATH_BAND
            : h->variant_on            ? AV_PATH_VARIANT
            : use_memo_rollout(h->cf)  ? AV_PATH_MEMO
            : use_env_warp_rollout(h->cf) ? AV_PATH_WARP
            : use_fast_rollout(h->cf)     ? AV_PATH_FAST
                                          : AV_PATH_BLOCK;
    return AV_OK;
}

int av_step_path(av_handle *h, int32_t *path)
{
    AV_HANDLE(h);
    if (!h || !path)
        return AV_EINVAL;
    if (h->large || h->variant_on || h->cf.path != 0)
        return av_rollout_path(h, path);  // av_step takes av_rollout's kernel
    *path = use_step_warp(h->cf) ? AV_PATH_STEP : AV_PATH_BLOCK;
    return AV_OK;
}

int av_warnings(av_handle *h, uint32_t *bits)
{
    AV_HANDLE(h);
    if (!h || !bits)
        return AV_EINVAL;
    AV_CUDA(h, cudaDeviceSynchronize());
    AV_CUDA(h, cudaMemcpy(bits, h->d_status + 1, 4, cudaMemcpyDeviceToHost));
    AV_CUDA(h, cudaMemset(h->d_status + 1, 0, 4));
    return AV_OK;
}

}  // extern "C"
