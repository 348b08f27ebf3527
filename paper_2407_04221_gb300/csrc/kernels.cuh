// kernels.cuh -- device code of libautoverse.so (sm_103a).
//
// State representation.  A board lives on chip as bit-planes: plane c holds
// channel c of every cell as a row-major bit string of H*W bits (cell p = y*W
// + x is bit p & 31 of word p >> 5).  Plane C is the transient force channel.
// Each plane word j is stored doubled as the pair (word j, word j+1), so any
// 32-bit window of a bit string is one 64-bit shared load plus one funnel
// shift.  A fused rollout keeps the planes resident for all its steps; cells
// are touched only when boards enter or leave the kernel.
//
// Matching (Sec. 2.1: a pattern matches where ReLU(conv_{K_I}(D) - I + 1) = 1,
// i.e. every present entry is set and, with absent entries as -1 weights,
// every absent entry is clear) is a bitwise AND over anchors: for anchor word
// a (anchors p = 32a .. 32a+31) and a term (channel c, window offset
// s = i*W + k), the anchors that pass are bits p + s of plane c.  One warp
// takes one rule; its four quarter-warps take the rule's four rotations (a
// rotation keeps the number of terms, so the quarters run the same loop), and
// lane q of a quarter owns anchor words q, q+8, q+16, ...  Terms are ordered
// so that the most selective come first; the warp leaves the rule as soon as
// no lane has a live anchor.  A live match pays the rule's reward per anchor
// and ORs the rule's output pattern into SET / CLEAR planes with shared
// atomics (the transposed-convolution write of Sec. 2.1).  Then
// next = (D & ~CLEAR) | (~D & SET), force dropped.
//
// Rule table layout (uint32 words; one table per env, or one shared):
//   [0] R   [1] total terms   [2] total outputs   [3] 0
//   [4 + 8r ...] rule r: n_present, n_absent, n_out, reward,
//                        first term, first output, shapes (rotation g in byte g:
//                        (h'-1)*5 + (w'-1)), 0
//   terms   (uint2, 16-byte aligned, [term][rotation]):
//           (byte offset of plane entry c*NWP + (s >> 5), s & 31 | kTermAbsent
//           for an absent term; funnel shifts use only the low five bits);
//           each rule's list is followed by padding terms up to a whole
//           number of kRestBatch terms after its first kRegTerms present ones,
//           and the table's list ends with one more batch of padding terms
//   outputs (uint4, [output][rotation]): (s >> 5, s & 31, set bits, clear bits)
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

namespace av {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kPlanePad = 10;   // zero entries past the last anchor slot of a plane
constexpr int kShapes = 25;     // (h', w') in 1..5 x 1..5
constexpr int kMaxCand = 4096;  // av_select: candidates per env
constexpr int kActChunk = 256;  // actions drawn ahead, per CTA
constexpr int kMaxSmemRuleWords = 8192;  // stage a rule table in shared memory up to 32 KiB
constexpr uint32_t kStatusVisitedOverflow = 1u;
constexpr uint32_t kStatusVisitedCount = 2u;  // a caller-owned visited count outside 0..capacity
constexpr uint32_t kWarnAction = 1u;
constexpr uint32_t kTermAbsent = 0x80000000u;  // flag in a term's shift word
// One warp per environment: present terms of a rule held in registers, and the
// batch in which the remaining terms are evaluated.  Each rule's term list is
// padded so that the terms after the register ones fill whole batches; a
// padding term reads plane C + 1 (the force of action 0, zero everywhere in
// that kernel's layout) as absent, so it passes.
constexpr int kRegTerms = 4;
constexpr int kRestBatch = 4;

struct DevConfig {
    int B, H, W, C, HW, NW, NWP, NA;  // NW plane words; NWP doubled entries per plane; NA words per lane
    int R, rules_per_env, max_steps, auto_reset;
    int ch_player, ch_goal, ch_empty, ch_wall, border_wall, cum_per_env;
    int cell_bytes;
    int rule_words;  // largest rule table (words) when tables are staged in shared memory, else 0
    int path;        // 0: choose; 1: block kernels; 2: fast rollout; 3: one warp per env; 4: memoising rollout
    int busy;        // rules expected to pass their register terms on most steps (host estimate)
    int fast_warps;  // fast rollout: warps per environment (4, or 8 when set to 8)
    int memo_stage;  // memo rollout: 0 the library decides, 1 rule tables in shared memory, 2 not
    int memo_warps;  // memo rollout: warps per environment (0: the default)
};

// Rule-table helpers shared by host (compiler) and device (reader).
__host__ __device__ inline uint32_t table_terms_word(int R) { return 4u + 8u * (uint32_t)R; }
__host__ __device__ inline uint32_t table_outs_word(int R, uint32_t total_terms)
{
    return table_terms_word(R) + 8u * total_terms;  // 4 rotations x uint2 per term
}

// ------------------------------------------------------------------ RNG
// SplitMix64 output finaliser (Vigna, splitmix64.c), keyed counter draw:
// draw(seed, st, a, b, c) = mix(mix(mix(seed + golden*(st+1)) ^ a) ^ (b<<32 | c)).
__device__ __forceinline__ uint64_t mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t draw(uint64_t seed, uint64_t st, uint64_t a, uint64_t b, uint64_t c)
{
    uint64_t z = mix64(seed + 0x9E3779B97F4A7C15ULL * (st + 1));
    z = mix64(z ^ a);
    return mix64(z ^ ((b << 32) | c));
}

__device__ __forceinline__ uint32_t uniform_below(uint64_t d, uint32_t n)
{
    return (uint32_t)(((d >> 32) * (uint64_t)n) >> 32);
}

// --------------------------------------------------------- shared memory
__host__ __device__ inline size_t align16(size_t x) { return (x + 15) & ~(size_t)15; }

struct StepSmem {
    size_t planes, setp, clrp, basep, vm, masks, red, acts, rules, cells, total;
};

// planes | SET | CLEAR | base planes (initial map, or a child) | valid-anchor
// masks [25][NW] | column masks [3][NW] | per-warp rewards + flags | cells
__host__ __device__ inline StepSmem step_smem(const DevConfig &cf, int n_cell_boards)
{
    StepSmem s;
    const size_t pw = (size_t)cf.C * cf.NW * 4;
    s.planes = 0;
    s.setp = align16((size_t)(cf.C + 1) * cf.NWP * 8);
    s.clrp = align16(s.setp + pw);
    s.basep = align16(s.clrp + pw);
    s.vm = align16(s.basep + pw);
    s.masks = align16(s.vm + (size_t)kShapes * cf.NW * 4);
    s.red = align16(s.masks + (size_t)3 * cf.NW * 4);
    s.acts = align16(s.red + (size_t)(kWarps + 16) * 4);
    s.rules = align16(s.acts + kActChunk);
    s.cells = align16(s.rules + (size_t)cf.rule_words * 4);
    s.total = align16(s.cells + (size_t)n_cell_boards * cf.HW * 2);
    return s;
}

struct Smem {
    uint2 *planes;
    uint32_t *setp, *clrp, *basep, *vm, *masks, *rules;
    int *red, *flags;  // flags: [0] a match this step, [1] action warning, [3] band step reward,
                       // [4] rollout_kernel's remembered actions, [5] its coming step's action,
                       // [6] the length of a run of repeated steps, [7] the action after a band
                       // kernel run, [8 + a] the remembered rewards
    uint8_t *acts;
    uint16_t *cells;
};

__device__ __forceinline__ Smem carve(unsigned char *smem, const DevConfig &cf, int n_cell_boards)
{
    const StepSmem L = step_smem(cf, n_cell_boards);
    Smem m;
    m.planes = reinterpret_cast<uint2 *>(smem + L.planes);
    m.setp = reinterpret_cast<uint32_t *>(smem + L.setp);
    m.clrp = reinterpret_cast<uint32_t *>(smem + L.clrp);
    m.basep = reinterpret_cast<uint32_t *>(smem + L.basep);
    m.vm = reinterpret_cast<uint32_t *>(smem + L.vm);
    m.masks = reinterpret_cast<uint32_t *>(smem + L.masks);
    m.red = reinterpret_cast<int *>(smem + L.red);
    m.flags = m.red + kWarps;
    m.acts = smem + L.acts;
    m.rules = reinterpret_cast<uint32_t *>(smem + L.rules);
    m.cells = reinterpret_cast<uint16_t *>(smem + L.cells);
    return m;
}

// Zero planes and SET/CLEAR, stage the anchor and column masks.
static __device__ void stage_common(const DevConfig &cf, const Smem &S, const uint32_t *__restrict__ vm_g,
                             const uint32_t *__restrict__ masks_g)
{
    const int tid = threadIdx.x;
    for (int i = tid; i < (cf.C + 1) * cf.NWP; i += kThreads)
        S.planes[i] = make_uint2(0u, 0u);
    for (int i = tid; i < cf.C * cf.NW; i += kThreads) {
        S.setp[i] = 0u;
        S.clrp[i] = 0u;
    }
    for (int i = tid; i < kShapes * cf.NW; i += kThreads)
        S.vm[i] = __ldg(vm_g + i);
    for (int i = tid; i < 3 * cf.NW; i += kThreads)
        S.masks[i] = __ldg(masks_g + i);
    if (tid < kWarps + 16)
        S.red[tid] = 0;
}

// Copy one env's rule table (n words, 16-byte aligned) into shared memory.
static __device__ void stage_rules(const uint32_t *__restrict__ tab, uint32_t n, uint32_t *dst)
{
    const uint4 *src = reinterpret_cast<const uint4 *>(tab);
    uint4 *d = reinterpret_cast<uint4 *>(dst);
    for (uint32_t i = threadIdx.x; i < n / 4; i += kThreads)
        d[i] = __ldg(src + i);
}

template <bool SM>
__device__ __forceinline__ uint4 ld4(const uint32_t *p)
{
    if (SM)
        return *reinterpret_cast<const uint4 *>(p);
    return __ldg(reinterpret_cast<const uint4 *>(p));
}

template <bool SM>
__device__ __forceinline__ uint2 ld2(const uint2 *p)
{
    if (SM)
        return *p;
    return __ldg(p);
}

// Write plane word w of channel c into the doubled layout.
// 64-bit shared load from a shared-window address.
__device__ __forceinline__ uint2 lds2(uint32_t addr)
{
    uint2 v;
    asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr));
    return v;
}

__device__ __forceinline__ void put_word(uint2 *planes, int NWP, int c, int w, uint32_t v)
{
    planes[c * NWP + w].x = v;
    if (w > 0)
        planes[c * NWP + w - 1].y = v;
}

// Board cells (global) -> tile planes: one warp ballot per channel per 32 cells.
// Writes the doubled planes when `dbl` is set, else plain words into `flat`.
template <typename CellT>
__device__ void cells_to_planes(const DevConfig &cf, const CellT *__restrict__ src, uint2 *dbl,
                                uint32_t *flat)
{
    const int tid = threadIdx.x, lane = tid & 31;
    for (int base = 0; base < cf.HW; base += kThreads) {
        const int p = base + tid;
        const uint32_t v = p < cf.HW ? (uint32_t)src[p] : 0u;
        const int w = p >> 5;  // warp-uniform
        for (int c = 0; c < cf.C; ++c) {
            const uint32_t bits = __ballot_sync(0xffffffffu, (v >> c) & 1u);
            if (lane == 0 && w < cf.NW) {
                if (dbl)
                    put_word(dbl, cf.NWP, c, w, bits);
                else
                    flat[c * cf.NW + w] = bits;
            }
        }
    }
}

// Cell p of a plane set (doubled or flat).
__device__ __forceinline__ uint32_t gather_cell(const DevConfig &cf, const uint2 *dbl,
                                                const uint32_t *flat, int p)
{
    const int w = p >> 5, b = p & 31;
    uint32_t v = 0;
    for (int c = 0; c < cf.C; ++c) {
        const uint32_t word = dbl ? dbl[c * cf.NWP + w].x : flat[c * cf.NW + w];
        v |= ((word >> b) & 1u) << c;
    }
    return v;
}

// Cells of a board from its doubled planes, stored to dst (global) a 32-bit
// word at a time by threads tid, tid + nthreads, ...: four 1-byte cells (bit k
// of a channel's 4-bit slice spread to byte k by a multiply) or two 2-byte
// cells.  Falls back to one cell per store when dst is not 4-byte aligned or
// the board does not fill whole words.
template <typename CellT>
__device__ __forceinline__ void store_cells(const DevConfig &cf, const uint2 *dbl, CellT *dst, int tid,
                                            int nthreads)
{
    constexpr int kPer = 4 / (int)sizeof(CellT);
    const int HW = cf.HW, NWP = cf.NWP;
    const int n_words = (HW + kPer - 1) / kPer;
    const bool aligned = (HW % kPer) == 0 && (reinterpret_cast<uintptr_t>(dst) & 3u) == 0;
    for (int g = tid; g < n_words; g += nthreads) {
        const int p0 = g * kPer, j = p0 >> 5, b = p0 & 31;
        uint32_t v = 0;
        for (int c = 0; c < cf.C; ++c) {
            const uint32_t x = dbl[c * NWP + j].x >> b;
            const uint32_t spread = sizeof(CellT) == 1 ? ((x & 0xfu) * 0x00204081u) & 0x01010101u
                                                       : ((x & 0x3u) * 0x00008001u) & 0x00010001u;
            v |= spread << c;
        }
        if (aligned) {
            reinterpret_cast<uint32_t *>(dst)[g] = v;
        } else {
            for (int k = 0; k < kPer && p0 + k < HW; ++k)
                dst[p0 + k] = (CellT)(v >> (8 * (int)sizeof(CellT) * k));
        }
    }
}

// The board's cells (from the doubled planes) into n consecutive steps of a
// trajectory: dst0, dst0 + stride, ... (stride in cells; each cell word built
// once).
template <typename CellT>
__device__ __forceinline__ void store_cells_steps(const DevConfig &cf, const uint2 *dbl, CellT *dst0, size_t stride,
                                                  int n, int tid, int nthreads)
{
    constexpr int kPer = 4 / (int)sizeof(CellT);
    const int HW = cf.HW, NWP = cf.NWP;
    const int n_words = (HW + kPer - 1) / kPer;
    const bool aligned = (HW % kPer) == 0 && (reinterpret_cast<uintptr_t>(dst0) & 3u) == 0 &&
                         (stride * sizeof(CellT)) % 4 == 0;
    for (int g = tid; g < n_words; g += nthreads) {
        const int p0 = g * kPer, j = p0 >> 5, b = p0 & 31;
        uint32_t v = 0;
        for (int c = 0; c < cf.C; ++c) {
            const uint32_t x = dbl[c * NWP + j].x >> b;
            const uint32_t spread = sizeof(CellT) == 1 ? ((x & 0xfu) * 0x00204081u) & 0x01010101u
                                                       : ((x & 0x3u) * 0x00008001u) & 0x00010001u;
            v |= spread << c;
        }
        for (int k = 0; k < n; ++k) {
            CellT *dst = dst0 + (size_t)k * stride;
            if (aligned) {
                reinterpret_cast<uint32_t *>(dst)[g] = v;
            } else {
                for (int i = 0; i < kPer && p0 + i < HW; ++i)
                    dst[p0 + i] = (CellT)(v >> (8 * (int)sizeof(CellT) * i));
            }
        }
    }
}

// Force plane for `action`, from the player plane (warp-cooperative, one warp).
// Player at p puts force at p + d: d = -W up, +1 right, +W down, -1 left,
// dropped where it would leave the board.
static __device__ void force_plane(const DevConfig &cf, uint2 *planes, const uint32_t *masks, int action)
{
    const int lane = threadIdx.x & 31, NW = cf.NW, NWP = cf.NWP;
    const uint32_t *firstcol = masks, *lastcol = masks + NW, *cellmask = masks + 2 * NW;
    const bool on = cf.ch_player >= 0 && action >= 1 && action <= 4;
    const uint2 *P = planes + (on ? cf.ch_player : 0) * NWP;
    for (int w = lane; w < NW; w += 32) {
        uint32_t f = 0;
        if (on) {
            const int n = (action == 1 || action == 3) ? cf.W : 1;
            const int q = n >> 5, r = n & 31;
            if (action == 1 || action == 4) {  // toward lower p: bits [32w + n, 32w + n + 32)
                const uint2 e = P[w + q];
                f = __funnelshift_r(e.x, e.y, r);
            } else {  // toward higher p: bits [32w - n, 32w - n + 32)
                const int j = w - q;
                if (j >= 1) {
                    const uint2 e = P[j - 1];
                    f = __funnelshift_l(e.x, e.y, r);
                } else if (j == 0) {
                    f = P[0].x << r;
                }
            }
            if (action == 2)
                f &= ~firstcol[w];
            else if (action == 4)
                f &= ~lastcol[w];
            f &= cellmask[w];
        }
        put_word(planes, NWP, cf.C, w, f);
    }
}

__device__ __forceinline__ void write_force(const DevConfig &cf, const Smem &S, int action)
{
    force_plane(cf, S.planes, S.masks, action);
}

// Force planes of actions a0, a0 + stride, ... < 5 from the player plane (one
// warp), into planes first + action.
static __device__ void force_planes(const DevConfig &cf, uint2 *P, const uint32_t *masks, int a0, int stride,
                                    int first)
{
    const int lane = threadIdx.x & 31, NW = cf.NW, NWP = cf.NWP;
    const uint32_t *firstcol = masks, *lastcol = masks + NW, *cellmask = masks + 2 * NW;
    const uint2 *pl = P + (cf.ch_player >= 0 ? cf.ch_player : 0) * NWP;
    for (int action = a0; action < 5; action += stride)
        for (int w = lane; w < NW; w += 32) {
            uint32_t f = 0;
            if (cf.ch_player >= 0 && action > 0) {
                const int n = (action == 1 || action == 3) ? cf.W : 1;
                const int q = n >> 5, r = n & 31;
                if (action == 1 || action == 4) {
                    const uint2 e = pl[w + q];
                    f = __funnelshift_r(e.x, e.y, r);
                } else {
                    const int j = w - q;
                    if (j >= 1) {
                        const uint2 e = pl[j - 1];
                        f = __funnelshift_l(e.x, e.y, r);
                    } else if (j == 0) {
                        f = pl[0].x << r;
                    }
                }
                if (action == 2)
                    f &= ~firstcol[w];
                else if (action == 4)
                    f &= ~lastcol[w];
                f &= cellmask[w];
            }
            put_word(P, NWP, first + action, w, f);
        }
}


__device__ __forceinline__ void scatter_bits(uint32_t *dst, uint32_t chans, int NW, int w0, uint32_t lo,
                                             uint32_t hi)
{
    while (chans) {
        const int c = __ffs(chans) - 1;
        chans &= chans - 1;
        if (lo)
            atomicOr(&dst[c * NW + w0], lo);
        if (hi)
            atomicOr(&dst[c * NW + w0 + 1], hi);
    }
}

// One warp evaluates rule r in its four rotations over every anchor; returns
// this lane's share of the reward and ORs the outputs of live matches into
// the SET / CLEAR planes.  Present terms AND in the window bits, absent terms
// AND in their complement; two terms per warp vote, and the warp leaves as
// soon as no lane has a live anchor.
template <int NA, bool SM>
__device__ __forceinline__ int match_rule(const DevConfig &cf, const uint32_t *tab, int r, const Smem &S)
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    const uint4 h0 = ld4<SM>(tab + 4 + 8 * r);  // n_present, n_absent, n_out, reward
    const uint4 h1 = ld4<SM>(tab + 8 + 8 * r);  // first term, first output, shapes
    const int shape = (int)((h1.z >> (8 * g)) & 0xffu);
    const uint32_t *vmr = S.vm + shape * cf.NW;
    uint32_t m[NA];
#pragma unroll
    for (int u = 0; u < NA; ++u) {
        const int a = q + 8 * u;
        m[u] = a < cf.NW ? vmr[a] : 0u;
    }
    const uint2 *tp = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R)) + (size_t)h1.x * 4 + g;
    const unsigned char *pb = reinterpret_cast<const unsigned char *>(S.planes) + q * 8;
    const uint32_t np = h0.x, nt = h0.x + h0.y;
    uint32_t t = 0;
    for (; t < nt; t += 2) {
        const bool two = t + 1 < nt && (t + 1 < np || t >= np);
        const uint32_t neg = t < np ? 0u : 0xffffffffu;
        const uint2 d0 = ld2<SM>(tp + 4 * t);
        const uint2 d1 = two ? ld2<SM>(tp + 4 * t + 4) : d0;
        uint32_t any = 0;
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            const uint2 w0 = *reinterpret_cast<const uint2 *>(pb + d0.x + 64 * u);
            const uint2 w1 = *reinterpret_cast<const uint2 *>(pb + d1.x + 64 * u);
            const uint32_t x0 = __funnelshift_r(w0.x, w0.y, d0.y) ^ neg;
            const uint32_t x1 = __funnelshift_r(w1.x, w1.y, d1.y) ^ neg;
            m[u] &= x0 & x1;
            any |= m[u];
        }
        if (!two)
            t -= 1;  // consumed one term
        if (!__any_sync(0xffffffffu, any != 0u))
            return 0;
    }
    uint32_t cnt = 0;
#pragma unroll
    for (int u = 0; u < NA; ++u)
        cnt += __popc(m[u]);
    if (cnt == 0)
        return 0;
    const uint4 *op = reinterpret_cast<const uint4 *>(tab + table_outs_word(cf.R, tab[1])) + (size_t)h1.y * 4 + g;
    for (uint32_t o = 0; o < h0.z; ++o) {
        const uint4 ov = SM ? op[4 * o] : __ldg(op + 4 * o);
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            if (!m[u])
                continue;
            const int w0 = q + 8 * u + (int)ov.x;
            const uint32_t lo = m[u] << ov.y;
            const uint32_t hi = ov.y ? (m[u] >> (32u - ov.y)) : 0u;
            scatter_bits(S.setp, ov.z, cf.NW, w0, lo, hi);
            scatter_bits(S.clrp, ov.w, cf.NW, w0, lo, hi);
        }
    }
    S.flags[0] = 1;
    return (int)h0.w * (int)cnt;
}

// All warps: every rule; per-warp reward sums land in S.red[warp].
template <int NA, bool SM>
__device__ __forceinline__ void match_all(const DevConfig &cf, const uint32_t *tab, const Smem &S)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int rew = 0;
    for (int r = warp; r < cf.R; r += kWarps)
        rew += match_rule<NA, SM>(cf, tab, r, S);
    rew = __reduce_add_sync(0xffffffffu, rew);
    if (lane == 0)
        S.red[warp] = rew;
}

__device__ __forceinline__ int action_at(const uint8_t *__restrict__ actions, uint64_t seed, int env, int s,
                                         int *warn_flag)
{
    int a = actions ? (int)actions[env] : (int)uniform_below(draw(seed, 4, (uint64_t)env, 0, (uint64_t)s), 5);
    if (a > 4) {
        *warn_flag = 1;
        a = 0;
    }
    return a;
}

// Actions of steps [s0, s0 + kActChunk) into the ring S.acts (one per thread).
__device__ __forceinline__ void fill_actions(const uint8_t *__restrict__ actions, uint64_t seed, int env, int s0,
                                             int n_steps, const Smem &S)
{
    const int s = s0 + (int)threadIdx.x;
    if (threadIdx.x < kActChunk && s < n_steps)
        S.acts[s & (kActChunk - 1)] = (uint8_t)action_at(actions, seed, env, s, S.flags + 1);
}

// ---------------------------------------------------------------- kernels
// Fused rollout (n_steps >= 1).  With `actions` non-null the action of step
// s is actions[env] (used by av_step, n_steps = 1); else it is drawn.
// SM: the env's rule table is staged in shared memory.  RUNS: runs of
// repeated steps are walked 32 at a time; the kernel of one-step launches
// leaves them out and keeps the compiler's own register choice (32 a thread
// for small boards), the others are held to 32 (small boards, eight CTAs per
// SM) or 64 registers.
template <typename CellT, int NA, bool SM, bool RUNS>
__global__ void __launch_bounds__(kThreads, RUNS ? (NA <= 2 ? 8 : 4) : 0)
rollout_kernel(DevConfig cf, const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
               const uint32_t *__restrict__ vm_g, const uint32_t *__restrict__ masks_g, CellT *cur,
               const CellT *__restrict__ init, int32_t *tsteps, int n_steps, uint64_t seed,
               const uint8_t *__restrict__ actions, CellT *obs_traj, int32_t *rew_traj,
               uint8_t *done_traj, int32_t *rew_sum, uint32_t *status)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const Smem S = carve(smem, cf, 0);
    const int env = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int HW = cf.HW, NW = cf.NW, NWP = cf.NWP, C = cf.C;
    const int table = cf.rules_per_env ? env : 0;
    const uint32_t *tab_g = arena + tab_off[table];
    const uint32_t *tab = SM ? S.rules : tab_g;

    stage_common(cf, S, vm_g, masks_g);
    if (SM)
        stage_rules(tab_g, tab_off[table + 1] - tab_off[table], S.rules);
    __syncthreads();
    cells_to_planes<CellT>(cf, cur + (size_t)env * HW, S.planes, nullptr);
    cells_to_planes<CellT>(cf, init + (size_t)env * HW, nullptr, S.basep);
    fill_actions(actions, seed, env, 0, n_steps, S);
    __syncthreads();

    int t = tsteps[env];
    int sum = 0;
    if (warp == 0) {
        write_force(cf, S, S.acts[0]);
        if (lane == 0)
            S.flags[5] = S.acts[0];  // the action of the coming step (the ring slot may be refilled)
    }
    __syncthreads();

    // While the board stays as it is, the step with action a always has the
    // same outcome: an action whose step matched nothing that changes the board
    // is remembered (bit a of S.flags[4], its reward in S.flags[8 + a]) and its
    // later steps skip the match; any change of the board forgets them all.
    for (int s = 0; s < n_steps; ++s) {
        const bool refill = ((s + 1) & (kActChunk - 1)) == 0;
        if (refill)
            fill_actions(actions, seed, env, s + 1, n_steps, S);
        // A run of repeated steps: from this step on, the steps whose actions
        // are remembered and that end no episode with an auto-reset take their
        // remembered rewards without a match or a board update, up to 32 at a
        // time (lane l of warp 0 takes step s + l) and never up to the last
        // step of the action ring's chunk (that step refills the ring).  Two
        // block barriers per run instead of two per step: the first publishes
        // the run's length once every warp has read this step's action; after
        // it warp 0 writes the next step's action and force plane, which the
        // second makes visible.
        if (RUNS && ((S.flags[4] >> S.flags[5]) & 1)) {  // block-uniform
            if (refill)
                __syncthreads();  // the ring's next chunk
            int a_next = 0;
            if (warp == 0) {
                const int lim = min(min(32, n_steps - s), ((s + 1) | (kActChunk - 1)) - s);
                const int a_l = lane == 0 ? S.flags[5] : lane < lim ? (int)S.acts[(s + lane) & (kActChunk - 1)] : 0;
                int goal = cf.ch_goal < 0;
                if (cf.ch_goal >= 0)
                    for (int w = lane; w < NW; w += 32)
                        goal |= S.planes[cf.ch_goal * NWP + w].x != 0u;
                goal = __any_sync(0xffffffffu, goal);
                const bool done_l = !goal || (cf.max_steps > 0 && t + lane + 1 >= cf.max_steps);
                const bool known_l = (S.flags[4] >> a_l) & 1;
                const uint32_t stop =
                    __ballot_sync(0xffffffffu, lane < lim && (!known_l || (done_l && cf.auto_reset)));
                const int e = stop ? __ffs(stop) - 1 : lim;  // steps s .. s + e - 1 repeat the board
                const int r_l = lane < e ? S.flags[8 + a_l] : 0;
                if (lane < e) {
                    if (rew_traj)
                        rew_traj[(size_t)(s + lane) * cf.B + env] = r_l;
                    if (done_traj)
                        done_traj[(size_t)(s + lane) * cf.B + env] = (uint8_t)done_l;
                }
                sum += __reduce_add_sync(0xffffffffu, r_l);
                t += e;
                a_next = __shfl_sync(0xffffffffu, a_l, e & 31);  // (read from the ring when e = lim)
                if (e == lim && s + e < n_steps)
                    a_next = S.acts[(s + e) & (kActChunk - 1)];
                if (lane == 0)
                    S.flags[6] = e;
            }
            __syncthreads();
            const int e = S.flags[6];
            if (e > 0) {
                if (warp == 0 && s + e < n_steps) {
                    write_force(cf, S, a_next);
                    if (lane == 0)
                        S.flags[5] = a_next;
                }
                if (obs_traj)
                    store_cells_steps<CellT>(cf, S.planes, obs_traj + ((size_t)s * cf.B + env) * HW,
                                             (size_t)cf.B * HW, e, tid, kThreads);
                __syncthreads();
                s += e - 1;
                continue;
            }
        }
        const int a = S.flags[5];
        const bool known = (S.flags[4] >> a) & 1;  // block-uniform (written before the last barrier)
        if (!known)
            match_all<NA, SM>(cf, tab, S);
        __syncthreads();
        if (warp == 0) {
            int rew, changed = 0;
            if (known) {
                rew = S.flags[8 + a];
            } else {
                rew = lane < kWarps ? S.red[lane] : 0;
                rew = __reduce_add_sync(0xffffffffu, rew);
                // combine: a bit changes where any match asks for it (one index over
                // every channel's words, so small boards keep all lanes busy)
                if (S.flags[0]) {
                    // (c, w) of index i = c * NW + w, stepped without a division
                    for (int i = lane, c = lane / NW, w = lane - (lane / NW) * NW; i < C * NW; i += 32) {
                        const uint32_t d = S.planes[c * NWP + w].x, st = S.setp[i], cl = S.clrp[i];
                        const uint32_t nd = (d & ~cl) | (~d & st);
                        S.setp[i] = 0u;
                        S.clrp[i] = 0u;
                        if (nd != d) {
                            changed = 1;
                            put_word(S.planes, NWP, c, w, nd);
                        }
                        for (w += 32; w >= NW; w -= NW)
                            ++c;
                    }
                    changed = __any_sync(0xffffffffu, changed);
                    __syncwarp();
                    if (lane == 0)
                        S.flags[0] = 0;
                }
                if (lane == 0) {  // remember the step: it left the board as it was
                    if (changed) {
                        S.flags[4] = 0;
                    } else {
                        S.flags[4] |= 1 << a;
                        S.flags[8 + a] = rew;
                    }
                }
            }
            int goal = cf.ch_goal < 0;
            if (cf.ch_goal >= 0)
                for (int w = lane; w < NW; w += 32)
                    goal |= S.planes[cf.ch_goal * NWP + w].x != 0u;
            goal = __any_sync(0xffffffffu, goal);
            t += 1;
            const int done = !goal || (cf.max_steps > 0 && t >= cf.max_steps);
            if (done && cf.auto_reset) {
                for (int i = lane, c = lane / NW, w = lane - (lane / NW) * NW; i < C * NW; i += 32) {
                    put_word(S.planes, NWP, c, w, S.basep[i]);
                    for (w += 32; w >= NW; w -= NW)
                        ++c;
                }
                t = 0;
                if (lane == 0)
                    S.flags[4] = 0;  // the board may have changed
            }
            sum += rew;
            if (lane == 0) {
                if (rew_traj)
                    rew_traj[(size_t)s * cf.B + env] = rew;
                if (done_traj)
                    done_traj[(size_t)s * cf.B + env] = (uint8_t)done;
            }
            __syncwarp();
            if (s + 1 < n_steps) {
                const int a_next = S.acts[(s + 1) & (kActChunk - 1)];
                write_force(cf, S, a_next);
                if (lane == 0)
                    S.flags[5] = a_next;
            }
        }
        __syncthreads();
        if (obs_traj) {
            store_cells<CellT>(cf, S.planes, obs_traj + ((size_t)s * cf.B + env) * HW, tid, kThreads);
        }
    }
    store_cells<CellT>(cf, S.planes, cur + (size_t)env * HW, tid, kThreads);
    if (tid == 0) {
        tsteps[env] = t;
        if (rew_sum)
            rew_sum[env] = sum;
        if (S.flags[1])
            atomicOr(status + 1, kWarnAction);
    }
}

// Tree-search expansion: one CTA per parent, the 5 children in turn.
template <typename CellT, int NA, bool SM>
__global__ void __launch_bounds__(kThreads)
expand_kernel(DevConfig cf, const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
              const uint32_t *__restrict__ vm_g, const uint32_t *__restrict__ masks_g,
              const CellT *__restrict__ parents, int F, const int32_t *__restrict__ n_parent,
              CellT *children, int32_t *rewards, uint8_t *done, uint64_t *hashes)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const Smem S = carve(smem, cf, 5);
    const int node = blockIdx.x, env = node / F, tid = threadIdx.x, warp = tid >> 5;
    const int HW = cf.HW, NW = cf.NW, NWP = cf.NWP, C = cf.C;
    if (n_parent && node - env * F >= n_parent[env])
        return;  // block-uniform: an empty frontier slot
    const int table = cf.rules_per_env ? env : 0;
    const uint32_t *tab_g = arena + tab_off[table];
    const uint32_t *tab = SM ? S.rules : tab_g;

    stage_common(cf, S, vm_g, masks_g);
    if (SM)
        stage_rules(tab_g, tab_off[table + 1] - tab_off[table], S.rules);
    __syncthreads();
    cells_to_planes<CellT>(cf, parents + (size_t)node * HW, S.planes, nullptr);
    __syncthreads();

    for (int a = 0; a < 5; ++a) {
        if (warp == 0)
            write_force(cf, S, a);
        __syncthreads();
        match_all<NA, SM>(cf, tab, S);
        __syncthreads();
        const int any = S.flags[0];
        for (int i = tid; i < C * NW; i += kThreads) {  // child planes
            const int c = i / NW, w = i - c * NW;
            const uint32_t d = S.planes[c * NWP + w].x;
            uint32_t v = d;
            if (any) {
                v = (d & ~S.clrp[i]) | (~d & S.setp[i]);
                S.setp[i] = 0u;
                S.clrp[i] = 0u;
            }
            S.basep[i] = v;
        }
        __syncthreads();
        uint16_t *cells = S.cells + (size_t)a * HW;
        CellT *dst = children + ((size_t)node * 5 + a) * HW;
        int goal = 0;
        for (int p = tid; p < HW; p += kThreads) {
            const uint32_t v = gather_cell(cf, nullptr, S.basep, p);
            cells[p] = (uint16_t)v;
            dst[p] = (CellT)v;
            if (cf.ch_goal >= 0)
                goal |= (int)((v >> cf.ch_goal) & 1u);
        }
        const int goal_left = __syncthreads_or(goal) || cf.ch_goal < 0;
        if (tid == 0) {
            int rew = 0;
            for (int w = 0; w < kWarps; ++w)
                rew += S.red[w];
            rewards[(size_t)node * 5 + a] = rew;
            if (done)
                done[(size_t)node * 5 + a] = (uint8_t)!goal_left;
            S.flags[0] = 0;
        }
    }
    __syncthreads();
    // FNV-1a 64 over the canonical bytes, one thread per child
    if ((tid & 31) == 0 && warp < 5) {
        const uint16_t *gc = S.cells + (size_t)warp * HW;
        uint64_t hsh = 0xcbf29ce484222325ULL;
        for (int p = 0; p < HW; ++p) {
            const uint32_t v = gc[p];
            hsh = (hsh ^ (v & 0xffu)) * 0x100000001b3ULL;
            if (sizeof(CellT) == 2)
                hsh = (hsh ^ (v >> 8)) * 0x100000001b3ULL;
        }
        hashes[(size_t)node * 5 + warp] = hsh;
    }
}

// ============================================================ warp-resident path
// Small boards (at most 16 plane words): one warp owns one environment for a
// whole launch, with its own planes, SET / CLEAR planes and staged rule table
// in shared memory.  It evaluates the first two terms of RB rules together
// (independent dependency chains), continues only the rules that still have a
// live anchor, and then updates its board itself: no block-wide barrier.

constexpr int kWarpCtaMax = 8;  // warps (= parents) per CTA at most

struct WarpSmem {
    uint2 *planes;
    uint32_t *setp, *clrp, *basep, *vm, *masks, *rules;
    uint8_t *acts;
    uint16_t *cells;
};

template <typename CellT>
__device__ void warp_cells_to_planes(const DevConfig &cf, const CellT *__restrict__ src, uint2 *dbl,
                                     uint32_t *flat)
{
    const int lane = threadIdx.x & 31;
    for (int base = 0; base < cf.HW; base += 32) {
        const int p = base + lane;
        const uint32_t v = p < cf.HW ? (uint32_t)src[p] : 0u;
        const int w = base >> 5;
        for (int c = 0; c < cf.C; ++c) {
            const uint32_t bits = __ballot_sync(0xffffffffu, (v >> c) & 1u);
            if (lane == 0) {
                if (dbl)
                    put_word(dbl, cf.NWP, c, w, bits);
                else
                    flat[c * cf.NW + w] = bits;
            }
        }
    }
}

// Shared memory of expand_warp_kernel: one region per CTA (the rule table when
// staged, valid-anchor masks, column masks), then per warp its planes, SET /
// CLEAR / child planes and the canonical bytes of its five children.  All
// warps of a CTA expand parents of one environment (the host makes the warp
// count divide F), so they share the table.
struct ExpandLayout {
    size_t vm, masks, rules, warps;  // CTA region
    size_t planes, setp, clrp, basep, bytes, per_warp;  // offsets within a warp's region
    size_t child_bytes;  // canonical bytes of one child, padded to 16
};

// Per warp: C tile planes and the force planes of the five actions (C + a),
// doubled; SET and CLEAR planes per action; the five children's canonical
// bytes.
__host__ __device__ inline ExpandLayout expand_layout(const DevConfig &cf)
{
    ExpandLayout L;
    const size_t pw = (size_t)cf.C * cf.NW * 4;
    L.vm = 0;
    L.masks = align16((size_t)kShapes * cf.NW * 4);
    L.rules = align16(L.masks + (size_t)3 * cf.NW * 4);
    L.warps = align16(L.rules + (size_t)cf.rule_words * 4);
    L.child_bytes = align16((size_t)cf.HW * cf.cell_bytes);
    L.planes = 0;
    L.setp = align16((size_t)(cf.C + 5) * cf.NWP * 8);
    L.clrp = align16(L.setp + 5 * pw);
    L.basep = L.clrp;  // not used
    L.bytes = align16(L.clrp + 5 * pw);
    L.per_warp = align16(L.bytes + 5 * L.child_bytes);
    return L;
}

// Cells of a child board, (D & ~CLEAR) | (~D & SET) from the parent's doubled
// planes and the child's SET / CLEAR planes, written as canonical bytes to
// `out` (shared, 16-byte aligned) and to `dst` (global),
// and whether any goal tile is left.  One warp; a 32-bit word per lane per
// pass: four 1-byte cells (bit k of a channel's 4-bit slice spread to byte k
// by a multiply) or two 2-byte cells.
template <typename CellT>
__device__ __forceinline__ int planes_to_cells(const DevConfig &cf, const uint2 *dbl, const uint32_t *setp,
                                               const uint32_t *clrp, uint32_t *out, CellT *dst)
{
    const int lane = threadIdx.x & 31, HW = cf.HW, NW = cf.NW, NWP = cf.NWP;
    constexpr int kPer = 4 / (int)sizeof(CellT);  // cells per 32-bit word
    const int n_words = (HW + kPer - 1) / kPer;
    const bool aligned = (HW % kPer) == 0 && (reinterpret_cast<uintptr_t>(dst) & 3u) == 0;
    int goal = 0;
    for (int g = lane; g < n_words; g += 32) {
        const int p0 = g * kPer, j = p0 >> 5, b = p0 & 31;
        uint32_t v = 0;
        for (int c = 0; c < cf.C; ++c) {
            const uint32_t d = dbl[c * NWP + j].x, st = setp[c * NW + j], cl = clrp[c * NW + j];
            const uint32_t x = ((d & ~cl) | (~d & st)) >> b;  // the child's word
            const uint32_t spread = sizeof(CellT) == 1 ? ((x & 0xfu) * 0x00204081u) & 0x01010101u
                                                       : ((x & 0x3u) * 0x00008001u) & 0x00010001u;
            v |= spread << c;
        }
        out[g] = v;
        if (cf.ch_goal >= 0)
            goal |= (int)(((v >> cf.ch_goal) & (sizeof(CellT) == 1 ? 0x01010101u : 0x00010001u)) != 0u);
        if (aligned) {
            reinterpret_cast<uint32_t *>(dst)[g] = v;
        } else {
            for (int k = 0; k < kPer && p0 + k < HW; ++k)
                dst[p0 + k] = (CellT)(v >> (8 * (int)sizeof(CellT) * k));
        }
    }
    return __any_sync(0xffffffffu, goal) || cf.ch_goal < 0;
}

// One parent's five children (one warp).  A parent's children differ only in
// the force plane, so each rule's terms on tile channels are evaluated once
// (pass 1, four terms per vote); a rule with anchors left then applies its
// force terms for all five actions at once (pass 2) and writes each action's
// outputs into that action's SET / CLEAR planes.
// A child board from its parent's canonical words: a child differs from its
// parent only where its SET / CLEAR words flip a bit, so each output word is
// the parent's (tile bits only), rebuilt by planes_to_cells' formula where the
// plane word under it has a flipped bit.  `parent` (global, 4-byte aligned,
// whole words) holds the parent's canonical words.  Writes `out` (shared) and
// `dst` (global, 4-byte aligned); returns whether any goal tile is left.  One
// warp; boards of at most 32 plane words.
template <typename CellT>
__device__ __forceinline__ int child_cells(const DevConfig &cf, const uint2 *dbl, const uint32_t *setp,
                                           const uint32_t *clrp, const uint32_t *parent, uint32_t *out, CellT *dst)
{
    const int lane = threadIdx.x & 31, HW = cf.HW, NW = cf.NW, NWP = cf.NWP;
    constexpr int kPer = 4 / (int)sizeof(CellT);  // cells per 32-bit word
    const int n_words = HW / kPer;
    uint32_t flip = 0, goal = 0;
    if (lane < NW) {
        for (int c = 0; c < cf.C; ++c) {
            const uint32_t d = dbl[c * NWP + lane].x, st = setp[c * NW + lane], cl = clrp[c * NW + lane];
            flip |= (d & cl) | (~d & st);
            if (c == cf.ch_goal)
                goal = (d & ~cl) | (~d & st);
        }
    }
    const uint32_t changed = __ballot_sync(0xffffffffu, flip != 0u);  // plane words with a flipped bit
    const int goal_left = cf.ch_goal < 0 || __any_sync(0xffffffffu, goal != 0u);
    const uint32_t tiles = ((1u << cf.C) - 1u) * (sizeof(CellT) == 1 ? 0x01010101u : 0x00010001u);
    for (int g = lane; g < n_words; g += 32) {
        const int p0 = g * kPer, j = p0 >> 5, b = p0 & 31;
        uint32_t v;
        if ((changed >> j) & 1u) {
            v = 0;
            for (int c = 0; c < cf.C; ++c) {
                const uint32_t d = dbl[c * NWP + j].x, st = setp[c * NW + j], cl = clrp[c * NW + j];
                const uint32_t x = ((d & ~cl) | (~d & st)) >> b;
                const uint32_t spread = sizeof(CellT) == 1 ? ((x & 0xfu) * 0x00204081u) & 0x01010101u
                                                           : ((x & 0x3u) * 0x00008001u) & 0x00010001u;
                v |= spread << c;
            }
        } else {
            v = __ldg(parent + g) & tiles;
        }
        out[g] = v;
        reinterpret_cast<uint32_t *>(dst)[g] = v;
    }
    return goal_left;
}

template <typename CellT, int NA, bool SM>
__device__ __forceinline__ void expand_rules(const DevConfig &cf, const uint32_t *tab, const WarpSmem &S,
                                             int (&rew)[5])
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    const int NW = cf.NW;
    const uint32_t plane_bytes = (uint32_t)cf.NWP * 8;
    const uint32_t force0 = (uint32_t)cf.C * plane_bytes, force_end = force0 + plane_bytes;
    const uint32_t pbase = (uint32_t)__cvta_generic_to_shared(S.planes) + q * 8;
    const uint2 *terms = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R));
    const uint32_t cnw = (uint32_t)cf.C * NW;
    for (int r = 0; r < cf.R; ++r) {
        const uint4 h0 = ld4<SM>(tab + 4 + 8 * r);
        const uint4 h1 = ld4<SM>(tab + 8 + 8 * r);
        const uint32_t *vmr = S.vm + ((h1.z >> (8 * g)) & 0xffu) * NW;
        uint32_t m[NA];
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            const int a = q + 8 * u;
            m[u] = a < NW ? vmr[a] : 0u;
        }
        const uint2 *tp = terms + (size_t)h1.x * 4 + g;
        const uint32_t nt = h0.x + h0.y;
        // pass 1: tile-channel terms (a force term, or one past the end, passes)
        bool live = __any_sync(0xffffffffu, (m[0] | (NA > 1 ? m[NA - 1] : 0u)) != 0u);
        for (uint32_t t = 0; live && t < nt; t += 4) {
            uint2 d[4];
            bool skip[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                d[j] = t + j < nt ? ld2<SM>(tp + 4 * (t + j)) : make_uint2(force0, 0u);
                skip[j] = d[j].x >= force0 && d[j].x < force_end;
            }
            uint32_t any = 0;
#pragma unroll
            for (int u = 0; u < NA; ++u) {
                uint32_t x = m[u];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint2 w = lds2(pbase + (skip[j] ? 0u : d[j].x) + 64 * u);
                    const uint32_t v = __funnelshift_r(w.x, w.y, d[j].y) ^ (uint32_t)((int32_t)d[j].y >> 31);
                    x &= skip[j] ? 0xffffffffu : v;
                }
                m[u] = x;
                any |= x;
            }
            live = __any_sync(0xffffffffu, any != 0u);
        }
        if (!live)
            continue;
        // pass 2: the force terms, for every action
        uint32_t ma[5][NA];
#pragma unroll
        for (int a = 0; a < 5; ++a)
#pragma unroll
            for (int u = 0; u < NA; ++u)
                ma[a][u] = m[u];
        for (uint32_t t = 0; t < nt; ++t) {
            const uint2 d = ld2<SM>(tp + 4 * t);
            if (d.x < force0 || d.x >= force_end)  // the same for every rotation
                continue;
            const uint32_t neg = (uint32_t)((int32_t)d.y >> 31);
#pragma unroll
            for (int a = 0; a < 5; ++a)
#pragma unroll
                for (int u = 0; u < NA; ++u) {
                    const uint2 w = lds2(pbase + d.x + (uint32_t)a * plane_bytes + 64 * u);
                    ma[a][u] &= __funnelshift_r(w.x, w.y, d.y) ^ neg;
                }
        }
        const uint4 *op = reinterpret_cast<const uint4 *>(tab + table_outs_word(cf.R, tab[1])) + (size_t)h1.y * 4 + g;
#pragma unroll
        for (int a = 0; a < 5; ++a) {
            uint32_t cnt = 0;
#pragma unroll
            for (int u = 0; u < NA; ++u)
                cnt += __popc(ma[a][u]);
            if (cnt == 0)
                continue;
            rew[a] += (int)h0.w * (int)cnt;
            for (uint32_t o = 0; o < h0.z; ++o) {
                const uint4 ov = SM ? op[4 * o] : __ldg(op + 4 * o);
#pragma unroll
                for (int u = 0; u < NA; ++u) {
                    if (!ma[a][u])
                        continue;
                    const int w0 = q + 8 * u + (int)ov.x;
                    const uint32_t lo = ma[a][u] << ov.y;
                    const uint32_t hi = ov.y ? (ma[a][u] >> (32u - ov.y)) : 0u;
                    scatter_bits(S.setp + a * cnw, ov.z, NW, w0, lo, hi);
                    scatter_bits(S.clrp + a * cnw, ov.w, NW, w0, lo, hi);
                }
            }
        }
    }
}

template <typename CellT, int NA, bool SM>
__global__ void __launch_bounds__(32 * kWarpCtaMax)
expand_warp_kernel(DevConfig cf, const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
                   const uint32_t *__restrict__ vm_g, const uint32_t *__restrict__ masks_g,
                   const CellT *__restrict__ parents, int F, const int32_t *__restrict__ n_parent,
                   CellT *children, int32_t *rewards, uint8_t *done, uint64_t *hashes)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const ExpandLayout L = expand_layout(cf);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    const long long first = (long long)blockIdx.x * nwarps;  // this CTA's first parent
    const long long node = first + warp;
    const long long total = (long long)cf.B * F;
    const int env0 = (int)(min(first, total - 1) / F);
    bool mine = node < total;  // this warp has a parent to expand
    const int env = mine ? (int)(node / F) : env0;
    if (mine && n_parent && (int)(node - (long long)env * F) >= n_parent[env])
        mine = false;  // an empty frontier slot
    const int HW = cf.HW, NW = cf.NW, NWP = cf.NWP, C = cf.C;

    // ---- the CTA's shared region
    uint32_t *vm = reinterpret_cast<uint32_t *>(smem + L.vm);
    uint32_t *masks = reinterpret_cast<uint32_t *>(smem + L.masks);
    uint32_t *rules = reinterpret_cast<uint32_t *>(smem + L.rules);
    const int table = cf.rules_per_env ? env0 : 0;
    const uint32_t *tab_g = arena + tab_off[table];
    for (int i = threadIdx.x; i < kShapes * NW; i += blockDim.x)
        vm[i] = __ldg(vm_g + i);
    for (int i = threadIdx.x; i < 3 * NW; i += blockDim.x)
        masks[i] = __ldg(masks_g + i);
    if (SM) {
        const uint32_t n = tab_off[table + 1] - tab_off[table];
        const uint4 *src = reinterpret_cast<const uint4 *>(tab_g);
        uint4 *d = reinterpret_cast<uint4 *>(rules);
        for (uint32_t i = threadIdx.x; i < n / 4; i += blockDim.x)
            d[i] = __ldg(src + i);
    }
    // ---- this warp's region
    unsigned char *wr = smem + L.warps + (size_t)warp * L.per_warp;
    WarpSmem S;
    S.planes = reinterpret_cast<uint2 *>(wr + L.planes);
    S.setp = reinterpret_cast<uint32_t *>(wr + L.setp);
    S.clrp = reinterpret_cast<uint32_t *>(wr + L.clrp);
    S.basep = reinterpret_cast<uint32_t *>(wr + L.basep);
    S.vm = vm;
    S.masks = masks;
    S.rules = rules;
    S.acts = nullptr;
    S.cells = nullptr;
    uint32_t *bytes = reinterpret_cast<uint32_t *>(wr + L.bytes);
    const uint32_t *tab = SM ? rules : tab_g;
    for (int i = lane; i < (C + 5) * NWP; i += 32)
        S.planes[i] = make_uint2(0u, 0u);
    for (int i = lane; i < 5 * C * NW; i += 32) {
        S.setp[i] = 0u;
        S.clrp[i] = 0u;
    }
    __syncthreads();  // the shared region

    if (mine) {
        warp_cells_to_planes<CellT>(cf, parents + (size_t)node * HW, S.planes, nullptr);
        __syncwarp();
        force_planes(cf, S.planes, S.masks, 0, 1, C);
        __syncwarp();
        int rew[5] = {0, 0, 0, 0, 0};
        expand_rules<CellT, NA, SM>(cf, tab, S, rew);
        __syncwarp();  // every lane's SET / CLEAR bits
        // children from the parent's words where the board and both pointers
        // allow whole-word access, else rebuilt from the planes
        const CellT *par = parents + (size_t)node * HW;
        const bool words = (HW * (int)sizeof(CellT)) % 4 == 0 && (reinterpret_cast<uintptr_t>(par) & 3u) == 0 &&
                           (reinterpret_cast<uintptr_t>(children) & 3u) == 0;
#pragma unroll
        for (int a = 0; a < 5; ++a) {
            CellT *dst = children + ((size_t)node * 5 + a) * HW;
            const int goal_left =
                words ? child_cells<CellT>(cf, S.planes, S.setp + a * C * NW, S.clrp + a * C * NW,
                                           reinterpret_cast<const uint32_t *>(par), bytes + a * (L.child_bytes / 4), dst)
                      : planes_to_cells<CellT>(cf, S.planes, S.setp + a * C * NW, S.clrp + a * C * NW,
                                               bytes + a * (L.child_bytes / 4), dst);
            const int r = __reduce_add_sync(0xffffffffu, rew[a]);
            if (lane == 0) {
                rewards[(size_t)node * 5 + a] = r;
                if (done)
                    done[(size_t)node * 5 + a] = (uint8_t)!goal_left;
            }
            __syncwarp();
        }
    }
    __syncthreads();  // every child's bytes

    // ---- FNV-1a 64 over each child's canonical bytes, one thread per child
    const int nbytes = HW * (int)sizeof(CellT);
    for (int t = threadIdx.x; t < 5 * nwarps; t += blockDim.x) {
        const int w = t / 5, a = t - 5 * w;
        const long long nd = first + w;
        if (nd >= total)
            continue;
        const int e = (int)(nd / F);
        if (n_parent && (int)(nd - (long long)e * F) >= n_parent[e])
            continue;
        const uint32_t *cb = reinterpret_cast<const uint32_t *>(smem + L.warps + (size_t)w * L.per_warp + L.bytes) +
                             a * (L.child_bytes / 4);
        uint64_t hsh = 0xcbf29ce484222325ULL;
        int k = 0;
        for (; k + 4 <= nbytes; k += 4) {
            const uint32_t x = cb[k >> 2];
            hsh = (hsh ^ (x & 0xffu)) * 0x100000001b3ULL;
            hsh = (hsh ^ ((x >> 8) & 0xffu)) * 0x100000001b3ULL;
            hsh = (hsh ^ ((x >> 16) & 0xffu)) * 0x100000001b3ULL;
            hsh = (hsh ^ (x >> 24)) * 0x100000001b3ULL;
        }
        if (k < nbytes) {
            const uint32_t x = cb[k >> 2];
            for (int r = 0; k + r < nbytes; ++r)
                hsh = (hsh ^ ((x >> (8 * r)) & 0xffu)) * 0x100000001b3ULL;
        }
        hashes[(size_t)nd * 5 + a] = hsh;
    }
}

// A lane's anchor words, passed by value (a register array would go to local
// memory through a call).
template <int NA>
struct Words {
    uint32_t v[NA];
};

// ============================================================ fast rollout
// Boards of at most 16 plane words.  One CTA per environment with NWARP warps;
// warp w owns rules w, w + NWARP, ... (at most RPW).
//
// Planes (doubled entries): 0..C-1 tile channels, then C..C+4 the force for
// actions 0..4 (rebuilt only when the board changes).  A step reads the force
// of its action by offsetting its force terms by action x plane size; the
// offset of the next step is loaded before the step's barrier.
//
// Each lane holds, per owned rule, the shared addresses, shifts and force
// flags of the rule's first two present terms for its anchor word, and the
// word's valid-anchor mask: a rule's per-step test is two 64-bit shared loads,
// two funnel shifts and one AND.  Rules still live after it continue in the
// general loop (four terms per warp vote).  A step in which no rule matches
// changes nothing but the step counter: every thread goes on after a single
// barrier.  Otherwise all warps combine the SET / CLEAR planes, test the goal,
// reset, and rebuild the force planes.

struct FastLayout {
    size_t planes, setp, clrp, basep, vm, masks, ctl, acts, rules, total;
};

__host__ __device__ inline FastLayout fast_layout(const DevConfig &cf)
{
    FastLayout L;
    const size_t pw = (size_t)cf.C * cf.NW * 4;
    L.planes = 0;
    L.setp = align16((size_t)(cf.C + 7) * cf.NWP * 8);
    L.clrp = align16(L.setp + pw);
    L.basep = align16(L.clrp + pw);
    L.vm = align16(L.basep + pw);
    L.masks = align16(L.vm + (size_t)kShapes * cf.NW * 4);
    L.ctl = align16(L.masks + (size_t)3 * cf.NW * 4);
    L.acts = align16(L.ctl + 16 * 4);
    L.rules = align16(L.acts + kActChunk);
    L.total = align16(L.rules + (size_t)cf.rule_words * 4);
    return L;
}

struct FastSmem {
    uint2 *planes;
    uint32_t *setp, *clrp, *basep, *vm, *masks, *rules;
    int *ctl;  // [0], [1] matches so far at even / odd steps; [2] reward of the step;
               // [3] warning
    uint8_t *acts;
};


// Terms t0.. of rule r, four per warp vote, then the rule's write.  `m` holds
// the live anchors so far; force terms read `fdelta` bytes past the action-0
// force plane.  Returns (this lane's reward, 1 if this lane matched).
template <int NA, bool SM>
__device__ __noinline__ int2 fast_rule_rest(const DevConfig &cf, const uint32_t *tab, const FastSmem &S, int r,
                                            uint32_t t0, uint32_t fdelta, Words<NA> mw)
{
    uint32_t *m = mw.v;
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    const uint4 h0 = ld4<SM>(tab + 4 + 8 * r);
    const uint4 h1 = ld4<SM>(tab + 8 + 8 * r);
    const uint32_t force0 = (uint32_t)(cf.C * cf.NWP * 8), force_end = force0 + (uint32_t)(cf.NWP * 8);
    const uint2 *tp = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R)) + (size_t)h1.x * 4 + g;
    const unsigned char *pb = reinterpret_cast<const unsigned char *>(S.planes) + q * 8;
    const uint32_t np = h0.x, nt = h0.x + h0.y;
    // a missing term reads the all-zero action-0 force plane, complemented: it passes
    for (uint32_t t = t0; t < nt; t += 4) {
        uint2 d[4];
        uint32_t neg[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t tt = t + j;
            if (tt < nt) {
                d[j] = ld2<SM>(tp + 4 * tt);
                if (d[j].x >= force0 && d[j].x < force_end)
                    d[j].x += fdelta;
                neg[j] = tt < np ? 0u : 0xffffffffu;
            } else {
                d[j] = make_uint2(force0, 0u);
                neg[j] = 0xffffffffu;
            }
        }
        uint32_t any = 0;
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            uint32_t x = m[u];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const uint2 w = *reinterpret_cast<const uint2 *>(pb + d[j].x + 64 * u);
                x &= __funnelshift_r(w.x, w.y, d[j].y) ^ neg[j];
            }
            m[u] = x;
            any |= x;
        }
        if (!__any_sync(0xffffffffu, any != 0u))
            return make_int2(0, 0);
    }
    uint32_t cnt = 0;
#pragma unroll
    for (int u = 0; u < NA; ++u)
        cnt += __popc(m[u]);
    if (cnt == 0)
        return make_int2(0, 0);
    const uint4 *op = reinterpret_cast<const uint4 *>(tab + table_outs_word(cf.R, tab[1])) + (size_t)h1.y * 4 + g;
    for (uint32_t o = 0; o < h0.z; ++o) {
        const uint4 ov = SM ? op[4 * o] : __ldg(op + 4 * o);
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            if (!m[u])
                continue;
            const int w0 = q + 8 * u + (int)ov.x;
            const uint32_t lo = m[u] << ov.y;
            const uint32_t hi = ov.y ? (m[u] >> (32u - ov.y)) : 0u;
            scatter_bits(S.setp, ov.z, cf.NW, w0, lo, hi);
            scatter_bits(S.clrp, ov.w, cf.NW, w0, lo, hi);
        }
    }
    return make_int2((int)h0.w * (int)cnt, 1);
}


// Per-lane register data of one owned rule.
template <int NA>
struct FastRule {
    uint32_t vm[NA];
    uint32_t a0, a1;  // shared addresses of terms 0 and 1 (force terms: the action-0 plane)
    uint32_t s0, s1;  // their shifts
    uint32_t f0, f1;  // 1 for a force term (offset by the step's action), else 0
};

template <typename CellT, int NA, int NWARP, int RPW, bool SM>
__global__ void __launch_bounds__(32 * NWARP, NWARP == 8 ? 4 : 7)
rollout_fast_kernel(DevConfig cf, const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
                    const uint32_t *__restrict__ vm_g, const uint32_t *__restrict__ masks_g, CellT *cur,
                    const CellT *__restrict__ init, int32_t *tsteps, int n_steps, uint64_t seed,
                    const uint8_t *__restrict__ actions, CellT *obs_traj, int32_t *rew_traj,
                    uint8_t *done_traj, int32_t *rew_sum, uint32_t *status)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const FastLayout L = fast_layout(cf);
    FastSmem S;
    S.planes = reinterpret_cast<uint2 *>(smem + L.planes);
    S.setp = reinterpret_cast<uint32_t *>(smem + L.setp);
    S.clrp = reinterpret_cast<uint32_t *>(smem + L.clrp);
    S.basep = reinterpret_cast<uint32_t *>(smem + L.basep);
    S.vm = reinterpret_cast<uint32_t *>(smem + L.vm);
    S.masks = reinterpret_cast<uint32_t *>(smem + L.masks);
    S.ctl = reinterpret_cast<int *>(smem + L.ctl);
    S.acts = smem + L.acts;
    S.rules = reinterpret_cast<uint32_t *>(smem + L.rules);

    const int env = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 3, q = lane & 7;
    const int HW = cf.HW, NW = cf.NW, NWP = cf.NWP, C = cf.C;
    const int table = cf.rules_per_env ? env : 0;
    const uint32_t *tab_g = arena + tab_off[table];
    const uint32_t *tab = SM ? S.rules : tab_g;
    const uint32_t plane_bytes = (uint32_t)NWP * 8;

    // ---- stage
    for (int i = tid; i < (C + 6) * NWP; i += 32 * NWARP)
        S.planes[i] = make_uint2(0u, 0u);
    for (int i = tid; i < C * NW; i += 32 * NWARP) {
        S.setp[i] = 0u;
        S.clrp[i] = 0u;
    }
    for (int i = tid; i < kShapes * NW; i += 32 * NWARP)
        S.vm[i] = __ldg(vm_g + i);
    for (int i = tid; i < 3 * NW; i += 32 * NWARP)
        S.masks[i] = __ldg(masks_g + i);
    if (SM) {
        const uint32_t n = tab_off[table + 1] - tab_off[table];
        const uint4 *src = reinterpret_cast<const uint4 *>(tab_g);
        uint4 *d = reinterpret_cast<uint4 *>(S.rules);
        for (uint32_t i = tid; i < n / 4; i += 32 * NWARP)
            d[i] = __ldg(src + i);
    }
    if (tid < 16)
        S.ctl[tid] = 0;
    __syncthreads();
    for (int k = tid; k < kActChunk; k += 32 * NWARP)
        if (k < n_steps)
            S.acts[k] = (uint8_t)action_at(actions, seed, env, k, S.ctl + 3);
    {
        const CellT *src = cur + (size_t)env * HW, *isrc = init + (size_t)env * HW;
        for (int base = 0; base < HW; base += 32 * NWARP) {
            const int p = base + tid;
            const uint32_t v = p < HW ? (uint32_t)src[p] : 0u;
            const uint32_t vi = p < HW ? (uint32_t)isrc[p] : 0u;
            const int w = p >> 5;
            for (int c = 0; c < C; ++c) {
                const uint32_t bits = __ballot_sync(0xffffffffu, (v >> c) & 1u);
                const uint32_t ibits = __ballot_sync(0xffffffffu, (vi >> c) & 1u);
                if (lane == 0 && w < NW) {
                    put_word(S.planes, NWP, c, w, bits);
                    S.basep[c * NW + w] = ibits;
                }
            }
        }
    }
    __syncthreads();
    force_planes(cf, S.planes, S.masks, warp, NWARP, cf.C);

    // ---- per-lane register data of the owned rules
    FastRule<NA> fr[RPW];
    uint32_t slow = 0;
    {
        const uint32_t base = (uint32_t)__cvta_generic_to_shared(S.planes) + q * 8;
        const uint32_t force0 = (uint32_t)C * plane_bytes;
        const uint2 *terms = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R));
#pragma unroll
        for (int k = 0; k < RPW; ++k) {
            const int r = warp + k * NWARP;
            FastRule<NA> &f = fr[k];
#pragma unroll
            for (int u = 0; u < NA; ++u)
                f.vm[u] = 0;
            f.a0 = f.a1 = base;
            f.s0 = f.s1 = 0;
            f.f0 = f.f1 = 0;
            if (r < cf.R) {
                const uint4 h0 = ld4<SM>(tab + 4 + 8 * r);
                const uint4 h1 = ld4<SM>(tab + 8 + 8 * r);
                const uint32_t *vmr = S.vm + ((h1.z >> (8 * g)) & 0xffu) * NW;
#pragma unroll
                for (int u = 0; u < NA; ++u) {
                    const int a = q + 8 * u;
                    f.vm[u] = a < NW ? vmr[a] : 0u;
                }
                if (h0.x >= 2) {
                    const uint2 d0 = ld2<SM>(terms + (size_t)h1.x * 4 + g);
                    const uint2 d1 = ld2<SM>(terms + (size_t)(h1.x + 1) * 4 + g);
                    f.a0 = base + d0.x;
                    f.a1 = base + d1.x;
                    f.s0 = d0.y;
                    f.s1 = d1.y;
                    f.f0 = d0.x >= force0 && d0.x < force0 + plane_bytes;
                    f.f1 = d1.x >= force0 && d1.x < force0 + plane_bytes;
                } else {
                    slow |= 1u << k;  // fewer than two present terms: the general loop from term 0
                }
            }
        }
    }
    int t = tsteps[env];
    int goal_left;
    {
        int gl = cf.ch_goal < 0;
        if (cf.ch_goal >= 0)
            for (int w = lane; w < NW; w += 32)
                gl |= S.planes[cf.ch_goal * NWP + w].x != 0u;
        goal_left = __syncthreads_or(gl);  // also publishes the force planes
    }

    int seen0 = 0, seen1 = 0, sum = 0;
    uint32_t fdelta = (uint32_t)S.acts[0] * plane_bytes;
    for (int s = 0; s < n_steps; ++s) {
        const int par = s & 1;
        // ---- first pair of every owned rule from registers
        uint32_t m[RPW][NA];
        uint32_t anyall = 0;
#pragma unroll
        for (int k = 0; k < RPW; ++k) {
            const FastRule<NA> &f = fr[k];
            const uint32_t a0 = f.a0 + f.f0 * fdelta, a1 = f.a1 + f.f1 * fdelta;
#pragma unroll
            for (int u = 0; u < NA; ++u) {
                const uint2 w0 = lds2(a0 + 64 * u), w1 = lds2(a1 + 64 * u);
                m[k][u] = f.vm[u] & __funnelshift_r(w0.x, w0.y, f.s0) & __funnelshift_r(w1.x, w1.y, f.s1);
                anyall |= m[k][u];
            }
        }
        if (__any_sync(0xffffffffu, anyall != 0u) || slow) {  // rare: some rule still live
            int2 acc = make_int2(0, 0);
#pragma unroll
            for (int k = 0; k < RPW; ++k) {
                const bool from0 = (slow >> k) & 1u;
                uint32_t any = 0;
                Words<NA> mw;
#pragma unroll
                for (int u = 0; u < NA; ++u) {
                    mw.v[u] = from0 ? fr[k].vm[u] : m[k][u];
                    any |= mw.v[u];
                }
                if (!__any_sync(0xffffffffu, any != 0u))
                    continue;
                const int2 o = fast_rule_rest<NA, SM>(cf, tab, S, warp + k * NWARP, from0 ? 0u : 2u, fdelta, mw);
                acc.x += o.x;
                acc.y |= o.y;
            }
            const int wrew = __reduce_add_sync(0xffffffffu, acc.x);
            if (__any_sync(0xffffffffu, acc.y != 0) && lane == 0) {
                atomicAdd(S.ctl + 2, wrew);
                atomicAdd(S.ctl + par, 1);  // read after this step's barrier, next written two steps on
            }
        }
        // actions [s + 128, s + 256) into ring slots no step in [s, s + 128) reads
        if (warp == NWARP - 1 && s > 0 && (s & (kActChunk / 2 - 1)) == 0)
            for (int k = lane; k < kActChunk / 2; k += 32)
                if (s + kActChunk / 2 + k < n_steps)
                    S.acts[(s + kActChunk / 2 + k) & (kActChunk - 1)] =
                        (uint8_t)action_at(actions, seed, env, s + kActChunk / 2 + k, S.ctl + 3);
        const uint32_t fdelta_next = (uint32_t)S.acts[(s + 1) & (kActChunk - 1)] * plane_bytes;
        __syncthreads();

        const int matches = S.ctl[par];
        t += 1;
        int done = !goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
        if (matches == (par ? seen1 : seen0) && !(done && cf.auto_reset)) {
            // nothing changed: no reward, same board
            if (tid == 0) {
                if (rew_traj)
                    rew_traj[(size_t)s * cf.B + env] = 0;
                if (done_traj)
                    done_traj[(size_t)s * cf.B + env] = (uint8_t)done;
            }
        } else {
            if (par)
                seen1 = matches;
            else
                seen0 = matches;
            // combine, all warps: a bit changes where any match asks for it; one
            // thread per word, so the goal test of the new board comes with it
            int gl = cf.ch_goal < 0;
            for (int i = tid; i < C * NW; i += 32 * NWARP) {
                const int c = i / NW, w = i - c * NW;
                uint32_t d = S.planes[c * NWP + w].x;
                const uint32_t st = S.setp[i], cl = S.clrp[i];
                if (st | cl) {
                    S.setp[i] = 0u;
                    S.clrp[i] = 0u;
                    d = (d & ~cl) | (~d & st);
                    put_word(S.planes, NWP, c, w, d);
                }
                if (c == cf.ch_goal)
                    gl |= d != 0u;
            }
            goal_left = __syncthreads_or(gl);
            done = !goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
            if (done && cf.auto_reset) {
                for (int i = tid; i < C * NW; i += 32 * NWARP) {
                    const int c = i / NW, w = i - c * NW;
                    put_word(S.planes, NWP, c, w, S.basep[i]);
                }
                t = 0;
                gl = cf.ch_goal < 0;
                if (cf.ch_goal >= 0)
                    for (int w = tid; w < NW; w += 32 * NWARP)
                        gl |= S.basep[cf.ch_goal * NW + w] != 0u;
                goal_left = __syncthreads_or(gl);
            }
            force_planes(cf, S.planes, S.masks, warp, NWARP, cf.C);
            if (tid == 0) {
                const int rew = S.ctl[2];
                sum += rew;
                S.ctl[2] = 0;
                if (rew_traj)
                    rew_traj[(size_t)s * cf.B + env] = rew;
                if (done_traj)
                    done_traj[(size_t)s * cf.B + env] = (uint8_t)done;
            }
            __syncthreads();
        }
        if (obs_traj) {
            store_cells<CellT>(cf, S.planes, obs_traj + ((size_t)s * cf.B + env) * HW, tid, 32 * NWARP);
        }
        fdelta = fdelta_next;
    }
    store_cells<CellT>(cf, S.planes, cur + (size_t)env * HW, tid, 32 * NWARP);
    if (tid == 0) {
        tsteps[env] = t;
        if (rew_sum)
            rew_sum[env] = sum;
        if (S.ctl[3])
            atomicOr(status + 1, kWarnAction);
    }
}

// ============================================================ one warp per environment
// Boards of at most 16 plane words and at most 16 rules.  A CTA holds
// blockDim.x / 32 environments, one warp each, every one with its own region
// of shared memory (FastLayout).  Planes: 0..C-1 tile channels, C the force of
// the current step, C+1..C+5 the force of actions 0..4 (rebuilt only when the
// board changes), C+6 all ones; the next step's force is copied into plane C
// at the end of each step.  Each lane keeps the first four present terms of
// every rule in registers (EnvRule; a rule with fewer reads the all-ones plane
// in their place), so a step in which no rule survives them is RPW x 4 shared
// loads, one vote and the force copy: no barrier, no shared counter.  Rules
// that do survive continue, one at a time, in a single inlined loop over the
// remaining terms (four per vote, the next four fetched ahead).  A rule that
// survives its register terms is first tested once per board on its tile
// terms alone (env_dead_rules): one that passes nowhere on them is left out,
// of the quiet loop's vote too, until the board changes, so that a rule stuck
// a term short of a match does not cost a general step every step.  A step
// with a match combines the SET / CLEAR planes, tests the goal, resets when due and
// rebuilds the five force planes, all within the warp.

// Per-lane register data of one rule: its valid anchors in this lane's words
// and the shared addresses and shifts of its first four present terms.
template <int NA>
struct EnvRule {
    uint32_t vm[NA];
    uint32_t a[kRegTerms], s[kRegTerms];
    uint32_t rest;  // the remaining terms: (first descriptor index for this lane's rotation) << 8 | batches
};

// Anchors of this lane's word u that pass the register-resident terms.
template <int NA>
__device__ __forceinline__ uint32_t env_reg_terms(const EnvRule<NA> &f, int u)
{
    uint32_t x = f.vm[u];
#pragma unroll
    for (int j = 0; j < kRegTerms; ++j) {
        const uint2 w = lds2(f.a[j] + 64 * u);
        x &= __funnelshift_r(w.x, w.y, f.s[j]);
    }
    return x;
}

// The terms of rule r after its register-resident ones, for one environment,
// then the rule's write.  `rest` locates those terms (EnvRule::rest); `m`
// holds the anchors live after the register terms; `pbase` is the shared
// address of this lane's word in plane 0.  Every
// remaining term is evaluated, kRestBatch per iteration (the padded list has
// whole batches) with the next batch's descriptors already loaded: a rule that
// gets this far usually has few live anchors, and a warp vote per few terms
// costs more than the terms it would skip.  Returns (this lane's reward, 1 if
// this lane matched).
template <int NA, bool SM>
__device__ __forceinline__ int2 env_rule_rest(const DevConfig &cf, const uint32_t *tab, uint32_t pbase,
                                              uint32_t *setp, uint32_t *clrp, int r, uint32_t rest,
                                              uint32_t (&m)[NA])
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    const uint2 *tp = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R)) + (rest >> 8);
    const uint32_t nb = rest & 0xffu;  // padded batches
    // the table ends its term list with a batch of passing terms, so a batch
    // read past this rule's last one stays inside the list
    uint2 dn[kRestBatch];
#pragma unroll
    for (int j = 0; j < kRestBatch; ++j)
        dn[j] = ld2<SM>(tp + 4 * j);
    for (uint32_t b = 0; b < nb; ++b) {
        uint2 d[kRestBatch];
        tp += 4 * kRestBatch;
#pragma unroll
        for (int j = 0; j < kRestBatch; ++j) {
            d[j] = dn[j];
            dn[j] = ld2<SM>(tp + 4 * j);
        }
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            uint32_t v[kRestBatch];
#pragma unroll
            for (int j = 0; j < kRestBatch; ++j) {
                const uint2 w = lds2(pbase + d[j].x + 64 * u);
                v[j] = __funnelshift_r(w.x, w.y, d[j].y) ^ (uint32_t)((int32_t)d[j].y >> 31);
            }
            // a balanced AND: the terms of a batch do not wait on one another
            uint32_t x = v[0];
#pragma unroll
            for (int j = 1; j < kRestBatch; ++j)
                x &= v[j];
            m[u] &= x;
        }
    }
    uint32_t cnt = 0;
#pragma unroll
    for (int u = 0; u < NA; ++u)
        cnt += __popc(m[u]);
    if (cnt == 0)
        return make_int2(0, 0);
    const uint4 h0 = ld4<SM>(tab + 4 + 8 * r);
    const uint4 h1 = ld4<SM>(tab + 8 + 8 * r);
    const uint4 *op = reinterpret_cast<const uint4 *>(tab + table_outs_word(cf.R, tab[1])) + (size_t)h1.y * 4 + g;
    for (uint32_t o = 0; o < h0.z; ++o) {
        const uint4 ov = SM ? op[4 * o] : __ldg(op + 4 * o);
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            if (!m[u])
                continue;
            const int w0 = q + 8 * u + (int)ov.x;
            const uint32_t lo = m[u] << ov.y;
            const uint32_t hi = ov.y ? (m[u] >> (32u - ov.y)) : 0u;
            scatter_bits(setp, ov.z, cf.NW, w0, lo, hi);
            scatter_bits(clrp, ov.w, cf.NW, w0, lo, hi);
        }
    }
    return make_int2((int)h0.w * (int)cnt, 1);
}

// A general step's per-step outputs (one warp): reward and done flag, and the
// board.  Not inlined: on one warp a branch around a large inline block costs
// tens of cycles even when not taken, around a call a few.
template <typename CellT>
__device__ __noinline__ void env_step_outputs(DevConfig cf, const uint2 *planes, int env, int s, int rew,
                                              int done, CellT *obs_traj, int32_t *rew_traj, uint8_t *done_traj)
{
    if ((threadIdx.x & 31) == 0) {
        if (rew_traj)
            rew_traj[(size_t)s * cf.B + env] = rew;
        if (done_traj)
            done_traj[(size_t)s * cf.B + env] = (uint8_t)done;
    }
    if (obs_traj)
        store_cells<CellT>(cf, planes, obs_traj + ((size_t)s * cf.B + env) * cf.HW, threadIdx.x & 31, 32);
}

// The board update of a general step in which a rule matched or a reset is
// due (one warp): combine (a bit changes where any match asks for it), goal
// test of the new board, auto-reset, the five force planes.  Returns (t,
// goal_left, done).  Not inlined, like env_step_outputs.
static __device__ __noinline__ int3 env_board_update(DevConfig cf, uint2 *planes, uint32_t *setp, uint32_t *clrp,
                                                     const uint32_t *basep, const uint32_t *masks, int t)
{
    const int lane = threadIdx.x & 31, C = cf.C, NW = cf.NW, NWP = cf.NWP;
    __syncwarp();  // every lane's SET / CLEAR bits
    int gl = cf.ch_goal < 0;
    for (int i = lane; i < C * NW; i += 32) {
        const int c = i / NW, w = i - c * NW;
        uint32_t d = planes[c * NWP + w].x;
        const uint32_t st = setp[i], cl = clrp[i];
        if (st | cl) {
            setp[i] = 0u;
            clrp[i] = 0u;
            d = (d & ~cl) | (~d & st);
            put_word(planes, NWP, c, w, d);
        }
        if (c == cf.ch_goal)
            gl |= d != 0u;
    }
    int goal_left = __any_sync(0xffffffffu, gl);
    int done = !goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
    if (done && cf.auto_reset) {
        for (int i = lane; i < C * NW; i += 32) {
            const int c = i / NW, w = i - c * NW;
            put_word(planes, NWP, c, w, basep[i]);
        }
        t = 0;
        gl = cf.ch_goal < 0;
        if (cf.ch_goal >= 0)
            for (int w = lane; w < NW; w += 32)
                gl |= basep[cf.ch_goal * NW + w] != 0u;
        goal_left = __any_sync(0xffffffffu, gl);
    }
    __syncwarp();  // the new board
    force_planes(cf, planes, masks, 0, 1, C + 1);
    __syncwarp();  // its force planes
    return make_int3(t, goal_left, done);
}

// Actions [s + 128, s + 256) into the ring slots of steps [s - 128, s), all
// read by now (one warp).  Not inlined, like env_step_outputs.
static __device__ __noinline__ void env_refill(const uint8_t *actions, uint64_t seed, int env, int s, int n_steps,
                                               uint8_t *acts, int *warn)
{
    const int lane = threadIdx.x & 31;
    for (int k = lane; k < kActChunk / 2; k += 32)
        if (s + kActChunk / 2 + k < n_steps)
            acts[(s + kActChunk / 2 + k) & (kActChunk - 1)] =
                (uint8_t)action_at(actions, seed, env, s + kActChunk / 2 + k, warn);
    __syncwarp();
}

// Anchors of this lane's words at which every tile-channel term of rule k
// passes on the current board (its force terms left out).  Only the force
// terms change from one step to the next while the board stays as it is.
template <int NA, bool SM>
__device__ __forceinline__ void env_tile_terms(const DevConfig &cf, const uint32_t *tab, const uint32_t *vm_s,
                                               uint32_t pbase, int k, uint32_t (&m)[NA])
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    const uint2 *terms = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R));
    const uint32_t plane_bytes = (uint32_t)cf.NWP * 8, force_lo = (uint32_t)cf.C * plane_bytes;
    const uint4 h0 = ld4<SM>(tab + 4 + 8 * k);
    const uint4 h1 = ld4<SM>(tab + 8 + 8 * k);
    const uint32_t *vmr = vm_s + ((h1.z >> (8 * g)) & 0xffu) * cf.NW;
#pragma unroll
    for (int u = 0; u < NA; ++u) {
        const int a = q + 8 * u;
        m[u] = a < cf.NW ? vmr[a] : 0u;
    }
    for (uint32_t j = 0; j < h0.x + h0.y; ++j) {
        const uint2 d = ld2<SM>(terms + (size_t)(h1.x + j) * 4 + g);
        if (d.x - force_lo < plane_bytes)
            continue;  // a force term
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            const uint2 w = lds2(pbase + d.x + 64 * u);
            m[u] &= __funnelshift_r(w.x, w.y, d.y) ^ (uint32_t)((int32_t)d.y >> 31);
        }
    }
}

// Of `rules` (a warp-uniform bit set), the rules whose tile-channel terms pass
// at no valid anchor of the current board (one warp): they cannot match again
// before the board changes.  Not inlined, like env_step_outputs: it runs
// once per rule and board.
template <int NA, bool SM>
static __device__ __noinline__ uint32_t env_dead_rules(DevConfig cf, const uint32_t *tab, const uint32_t *vm_s,
                                                       uint32_t pbase, uint32_t rules)
{
    uint32_t dead = 0;
    while (rules) {
        const int k = __ffs(rules) - 1;
        rules &= rules - 1;
        uint32_t m[NA], any = 0;
        env_tile_terms<NA, SM>(cf, tab, vm_s, pbase, k, m);
#pragma unroll
        for (int u = 0; u < NA; ++u)
            any |= m[u];
        if (!__any_sync(0xffffffffu, any != 0u))
            dead |= 1u << k;
    }
    return dead;
}

template <typename CellT, int NA, int RPW, bool SM>
__global__ void __launch_bounds__(128)
rollout_env_warp_kernel(DevConfig cf, const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
                        const uint32_t *__restrict__ vm_g, const uint32_t *__restrict__ masks_g, CellT *cur,
                        const CellT *__restrict__ init, int32_t *tsteps, int n_steps, uint64_t seed,
                        const uint8_t *__restrict__ actions, CellT *obs_traj, int32_t *rew_traj,
                        uint8_t *done_traj, int32_t *rew_sum, uint32_t *status)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const FastLayout L = fast_layout(cf);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    const int env = blockIdx.x * (blockDim.x >> 5) + warp;
    if (env >= cf.B)
        return;  // whole warp; the kernel has no block-wide barrier
    unsigned char *mine = smem + (size_t)warp * L.total;
    FastSmem S;
    S.planes = reinterpret_cast<uint2 *>(mine + L.planes);
    S.setp = reinterpret_cast<uint32_t *>(mine + L.setp);
    S.clrp = reinterpret_cast<uint32_t *>(mine + L.clrp);
    S.basep = reinterpret_cast<uint32_t *>(mine + L.basep);
    S.vm = reinterpret_cast<uint32_t *>(mine + L.vm);
    S.masks = reinterpret_cast<uint32_t *>(mine + L.masks);
    S.ctl = reinterpret_cast<int *>(mine + L.ctl);
    S.acts = mine + L.acts;
    S.rules = reinterpret_cast<uint32_t *>(mine + L.rules);

    const int HW = cf.HW, NW = cf.NW, NWP = cf.NWP, C = cf.C;
    const int table = cf.rules_per_env ? env : 0;
    const uint32_t *tab_g = arena + tab_off[table];
    const uint32_t *tab = SM ? S.rules : tab_g;
    const uint32_t plane_bytes = (uint32_t)NWP * 8;
    const uint32_t ones = (uint32_t)(C + 6) * plane_bytes;  // every bit set
    uint2 *const slot = S.planes + C * NWP;
    const uint2 *const fplanes = S.planes + (C + 1) * NWP;

    // ---- stage (this warp's environment only)
    for (int i = lane; i < (C + 7) * NWP; i += 32)
        S.planes[i] = i < (C + 6) * NWP ? make_uint2(0u, 0u) : make_uint2(0xffffffffu, 0xffffffffu);
    for (int i = lane; i < C * NW; i += 32) {
        S.setp[i] = 0u;
        S.clrp[i] = 0u;
    }
    for (int i = lane; i < kShapes * NW; i += 32)
        S.vm[i] = __ldg(vm_g + i);
    for (int i = lane; i < 3 * NW; i += 32)
        S.masks[i] = __ldg(masks_g + i);
    if (SM) {
        const uint32_t n = tab_off[table + 1] - tab_off[table];
        const uint4 *src = reinterpret_cast<const uint4 *>(tab_g);
        uint4 *d = reinterpret_cast<uint4 *>(S.rules);
        for (uint32_t i = lane; i < n / 4; i += 32)
            d[i] = __ldg(src + i);
    }
    if (lane < 16)
        S.ctl[lane] = 0;
    for (int k = lane; k < kActChunk; k += 32)  // every slot holds an action in 0..4
        S.acts[k] = k < n_steps ? (uint8_t)action_at(actions, seed, env, k, S.ctl + 3) : (uint8_t)0;
    __syncwarp();
    {
        const CellT *src = cur + (size_t)env * HW, *isrc = init + (size_t)env * HW;
        for (int base = 0; base < HW; base += 32) {
            const int p = base + lane;
            const uint32_t v = p < HW ? (uint32_t)src[p] : 0u;
            const uint32_t vi = p < HW ? (uint32_t)isrc[p] : 0u;
            const int w = p >> 5;
            for (int c = 0; c < C; ++c) {
                const uint32_t bits = __ballot_sync(0xffffffffu, (v >> c) & 1u);
                const uint32_t ibits = __ballot_sync(0xffffffffu, (vi >> c) & 1u);
                if (lane == 0 && w < NW) {
                    put_word(S.planes, NWP, c, w, bits);
                    S.basep[c * NW + w] = ibits;
                }
            }
        }
    }
    __syncwarp();
    force_planes(cf, S.planes, S.masks, 0, 1, C + 1);
    __syncwarp();
    if (lane < NW)
        slot[lane] = fplanes[S.acts[0] * NWP + lane];

    // ---- per-lane register data of every rule
    EnvRule<NA> fr[RPW];
    const uint32_t pbase = (uint32_t)__cvta_generic_to_shared(S.planes) + q * 8;
    {
        const uint2 *terms = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R));
#pragma unroll
        for (int k = 0; k < RPW; ++k) {
            EnvRule<NA> &f = fr[k];
#pragma unroll
            for (int u = 0; u < NA; ++u)
                f.vm[u] = 0;
#pragma unroll
            for (int j = 0; j < kRegTerms; ++j) {
                f.a[j] = pbase + ones;
                f.s[j] = 0;
            }
            f.rest = 0;
            if (k < cf.R) {
                const uint4 h0 = ld4<SM>(tab + 4 + 8 * k);
                const uint4 h1 = ld4<SM>(tab + 8 + 8 * k);
                const uint32_t *vmr = S.vm + ((h1.z >> (8 * g)) & 0xffu) * NW;
#pragma unroll
                for (int u = 0; u < NA; ++u) {
                    const int a = q + 8 * u;
                    f.vm[u] = a < NW ? vmr[a] : 0u;
                }
#pragma unroll
                for (int j = 0; j < kRegTerms; ++j)
                    if ((uint32_t)j < h0.x) {  // present terms lead the rule's term list
                        const uint2 d = ld2<SM>(terms + (size_t)(h1.x + j) * 4 + g);
                        f.a[j] = pbase + d.x;
                        f.s[j] = d.y;
                    }
                const uint32_t t0 = min(h0.x, (uint32_t)kRegTerms);
                const uint32_t nb = (h0.x + h0.y - t0 + kRestBatch - 1) / kRestBatch;  // padded batches
                f.rest = (((h1.x + t0) * 4 + g) << 8) | nb;
            }
        }
    }
    int t = tsteps[env];
    int goal_left;
    {
        int gl = cf.ch_goal < 0;
        if (cf.ch_goal >= 0)
            for (int w = lane; w < NW; w += 32)
                gl |= S.planes[cf.ch_goal * NWP + w].x != 0u;
        goal_left = __any_sync(0xffffffffu, gl);
    }
    __syncwarp();  // the force of step 0
    const bool traj = rew_traj != nullptr || done_traj != nullptr;

    int sum = 0;
    uint32_t m[RPW][NA];  // anchors of each rule live after its register terms
    // Rules already tested on the current board, and those of them that cannot
    // match on it (env_dead_rules; warp-uniform, cleared when the board
    // changes), and per rule a mask that is zero for such a rule, which the
    // quiet loop applies to its vote.  Kernels with more than eight rules per
    // lane run without the test: their registers are full already.
    constexpr bool kDeadTest = RPW <= 8;
    uint32_t known = 0, dead = 0;
    uint32_t alive[kDeadTest ? RPW : 1];
#pragma unroll
    for (int k = 0; k < (kDeadTest ? RPW : 1); ++k)
        alive[k] = 0xffffffffu;
    // Steps in which no rule survives its register terms and no reset is due:
    // t advances, the next step's force goes into the slot, nothing else
    // changes.  The loop is kept free of branches around rarely used code,
    // which cost tens of cycles each even when not taken.  Leaves s at the
    // first step it does not finish (lim at the latest), with that step's
    // register masks in m when s < lim.
    auto quiet_steps = [&](int &s, int lim, auto traj_tag) {
        constexpr bool TRAJ = decltype(traj_tag)::value;
        while (s < lim) {
            const int a_next = S.acts[(s + 1) & (kActChunk - 1)];
            const uint2 f_next = lane < NW ? fplanes[a_next * NWP + lane] : make_uint2(0u, 0u);
            uint32_t anyall = 0;
#pragma unroll
            for (int k = 0; k < RPW; ++k)
#pragma unroll
                for (int u = 0; u < NA; ++u) {
                    m[k][u] = env_reg_terms(fr[k], u);
                    anyall |= m[k][u] & alive[kDeadTest ? k : 0];
                }
            const bool reset_due = cf.auto_reset && !(goal_left && (cf.max_steps <= 0 || t + 1 < cf.max_steps));
            if (__any_sync(0xffffffffu, anyall != 0u) || reset_due)
                return;  // the general step takes it
            t += 1;
            if (TRAJ) {
                const int done = !goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
                if (lane == 0) {
                    if (rew_traj)
                        rew_traj[(size_t)s * cf.B + env] = 0;
                    if (done_traj)
                        done_traj[(size_t)s * cf.B + env] = (uint8_t)done;
                }
                if (obs_traj)
                    store_cells<CellT>(cf, S.planes, obs_traj + ((size_t)s * cf.B + env) * HW, lane, 32);
            }
            if (lane < NW)
                slot[lane] = f_next;  // every read of this step's force is behind the vote
            __syncwarp();
            ++s;
        }
    };
    const bool any_traj = traj || obs_traj != nullptr;
    int refilled = 0;
    for (int s = 0; s < n_steps;) {
        // actions [s + 128, s + 256) into the ring slots of steps [s - 128, s),
        // all read by now
        if (s > 0 && (s & (kActChunk / 2 - 1)) == 0 && s != refilled) {
            env_refill(actions, seed, env, s, n_steps, S.acts, S.ctl + 3);
            refilled = s;
        }
        const int lim = min(n_steps, ((s / (kActChunk / 2)) + 1) * (kActChunk / 2));
        if (any_traj)
            quiet_steps(s, lim, std::integral_constant<bool, true>());
        else
            quiet_steps(s, lim, std::integral_constant<bool, false>());
        if (s >= lim)
            continue;  // the end, or the next refill

        // ---- busy steps: while some rule passes its register terms (or a
        // reset is due) every step is a general step; their own loop, so that
        // a run of them does not leave and re-enter the quiet loop each step.
        // The first recomputes what the quiet loop stopped at.
        while (s < lim) {
            const int a_next = S.acts[(s + 1) & (kActChunk - 1)];
            uint2 f_next = lane < NW ? fplanes[a_next * NWP + lane] : make_uint2(0u, 0u);
            uint32_t bits = 0;
#pragma unroll
            for (int k = 0; k < RPW; ++k) {
                uint32_t a = 0;
#pragma unroll
                for (int u = 0; u < NA; ++u) {
                    m[k][u] = env_reg_terms(fr[k], u);
                    a |= m[k][u];
                }
                bits |= (a != 0u ? 1u : 0u) << k;
            }
            const uint32_t raw = __reduce_or_sync(0xffffffffu, bits);  // rules live past their register terms
            const bool reset_due = cf.auto_reset && !(goal_left && (cf.max_steps <= 0 || t + 1 < cf.max_steps));
            if (!raw && !reset_due)
                break;  // a quiet step: back to the quiet loop
            if (kDeadTest && (raw & ~known)) {  // rules live for the first time on this board
                dead |= env_dead_rules<NA, SM>(cf, tab, S.vm, pbase, raw & ~known);
                known |= raw;
#pragma unroll
                for (int k = 0; k < (kDeadTest ? RPW : 1); ++k)
                    alive[k] = ((dead >> k) & 1u) ? 0u : 0xffffffffu;
            }
            uint32_t live = raw & ~dead;
            if (!live && !reset_due)
                break;  // only rules that cannot match: the quiet loop takes this step

            // ---- general step s: the rest of every live rule, writes
            int rew = 0, changed = 0;
            if (live) {
                int2 acc = make_int2(0, 0);
                while (live) {
                    const int k = __ffs(live) - 1;
                    live &= live - 1;
                    uint32_t mk[NA], rk = 0;
#pragma unroll
                    for (int u = 0; u < NA; ++u)
                        mk[u] = 0;
#pragma unroll
                    for (int kk = 0; kk < RPW; ++kk)
                        if (kk == k) {
#pragma unroll
                            for (int u = 0; u < NA; ++u)
                                mk[u] = m[kk][u];
                            rk = fr[kk].rest;
                        }
                    const int2 o = env_rule_rest<NA, SM>(cf, tab, pbase, S.setp, S.clrp, k, rk, mk);
                    acc.x += o.x;
                    acc.y |= o.y;
                }
                rew = __reduce_add_sync(0xffffffffu, acc.x);
                changed = __any_sync(0xffffffffu, acc.y != 0);
            }

            t += 1;
            int done = !goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
            if (changed || (done && cf.auto_reset)) {
                const int3 r = env_board_update(cf, S.planes, S.setp, S.clrp, S.basep, S.masks, t);
                t = r.x;
                goal_left = r.y;
                done = r.z;
                f_next = lane < NW ? fplanes[a_next * NWP + lane] : make_uint2(0u, 0u);
                sum += rew;
                known = 0;  // a new board
                dead = 0;
#pragma unroll
                for (int k = 0; k < (kDeadTest ? RPW : 1); ++k)
                    alive[k] = 0xffffffffu;
            }
            // every read of this step's force is behind the step's last vote
            if (lane < NW)
                slot[lane] = f_next;
            __syncwarp();
            if (any_traj)
                env_step_outputs<CellT>(cf, S.planes, env, s, rew, done, obs_traj, rew_traj, done_traj);
            ++s;
        }
    }
    store_cells<CellT>(cf, S.planes, cur + (size_t)env * HW, lane, 32);
    if (lane == 0) {
        tsteps[env] = t;
        if (rew_sum)
            rew_sum[env] = sum;
        if (S.ctl[3])
            atomicOr(status + 1, kWarnAction);
    }
}

template <typename CellT>
__global__ void __launch_bounds__(kThreads)
reset_kernel(DevConfig cf, const uint32_t *__restrict__ cum_all, uint64_t seed, CellT *cur,
             CellT *init, int32_t *tsteps, CellT *obs)
{
    extern __shared__ __align__(16) unsigned char smem[];
    uint16_t *G = reinterpret_cast<uint16_t *>(smem);
    const int env = blockIdx.x, tid = threadIdx.x, HW = cf.HW, H = cf.H, W = cf.W, C = cf.C;
    const uint32_t *cum = cum_all + (size_t)(cf.cum_per_env ? env : 0) * C;
    for (int p = tid; p < HW; p += blockDim.x) {
        const int y = p / W, x = p - y * W;
        const bool border = y == 0 || y == H - 1 || x == 0 || x == W - 1;
        uint32_t v;
        if (cf.border_wall && border) {
            v = cf.ch_wall >= 0 ? 1u << cf.ch_wall : 0u;
        } else {
            const uint32_t u = (uint32_t)(draw(seed, 1, (uint64_t)env, (uint64_t)y, (uint64_t)x) >> 40);
            int t = 0;
            while (t < C - 1 && !(u < __ldg(cum + t)))
                ++t;
            v = 1u << t;
        }
        G[p] = (uint16_t)v;
    }
    __syncthreads();
    if (cf.ch_player >= 0 && tid < 32) {
        const int lane = tid;
        const uint64_t d = draw(seed, 2, (uint64_t)env, 0, 0);
        // floor cells, in row-major order
        int n_empty = 0;
        if (cf.ch_empty >= 0)
            for (int base = 0; base < HW; base += 32) {
                const int p = base + lane;
                n_empty += __popc(__ballot_sync(0xffffffffu, p < HW && ((G[p] >> cf.ch_empty) & 1u)));
            }
        int chosen = -1;
        for (int pass = 0; pass < 2 && chosen < 0; ++pass) {
            // pass 0: k-th floor cell; pass 1 (no floor): k-th interior cell
            int n = n_empty;
            if (pass == 0 && n_empty == 0)
                continue;
            if (pass == 1) {
                if (n_empty > 0)
                    break;
                n = 0;
                for (int base = 0; base < HW; base += 32) {
                    const int p = base + lane;
                    const int y = p / W, x = p - y * W;
                    const bool border = y == 0 || y == H - 1 || x == 0 || x == W - 1;
                    n += __popc(__ballot_sync(0xffffffffu, p < HW && !(cf.border_wall && border)));
                }
                if (n == 0)
                    break;
            }
            int k = (int)uniform_below(d, (uint32_t)n);
            for (int base = 0; base < HW && chosen < 0; base += 32) {
                const int p = base + lane;
                bool pred;
                if (pass == 0) {
                    pred = p < HW && ((G[p] >> cf.ch_empty) & 1u);
                } else {
                    const int y = p / W, x = p - y * W;
                    const bool border = y == 0 || y == H - 1 || x == 0 || x == W - 1;
                    pred = p < HW && !(cf.border_wall && border);
                }
                uint32_t m = __ballot_sync(0xffffffffu, pred);
                const int c = __popc(m);
                if (k < c) {
                    for (int j = 0; j < k; ++j)
                        m &= m - 1;
                    chosen = base + __ffs(m) - 1;
                } else {
                    k -= c;
                }
            }
        }
        if (lane == 0 && chosen >= 0)
            G[chosen] = (uint16_t)(G[chosen] | (1u << cf.ch_player));
    }
    __syncthreads();
    CellT *dc = cur + (size_t)env * HW, *di = init + (size_t)env * HW;
    CellT *dobs = obs ? obs + (size_t)env * HW : nullptr;
    for (int p = tid; p < HW; p += blockDim.x) {
        const CellT v = (CellT)G[p];
        dc[p] = v;
        di[p] = v;
        if (dobs)
            dobs[p] = v;
    }
    if (tid == 0)
        tsteps[env] = 0;
}

// --------------------------------------------------------------- search
struct Key128 {
    uint64_t hi, lo;
};

__device__ __forceinline__ bool key_less(const Key128 &a, const Key128 &b)
{
    return a.hi < b.hi || (a.hi == b.hi && a.lo < b.lo);
}

// One compare-exchange of a bitonic stage (block k, partner distance j): keys
// i and i ^ j, ascending where bit k of i is clear.
__device__ __forceinline__ void bitonic_cmpx(Key128 *keys, int i, int k, int j)
{
    const int ixj = i | j;
    const bool up = (i & k) == 0;
    const Key128 x = keys[i], y = keys[ixj];
    if (key_less(y, x) == up) {
        keys[i] = y;
        keys[ixj] = x;
    }
}

// Lower key of the p-th compare-exchange pair of stage distance j within the
// 64-key chunk c.
__device__ __forceinline__ int bitonic_pair(int c, int p, int j)
{
    return (c << 6) | ((p & ~(j - 1)) << 1) | (p & (j - 1));
}

// Block-wide bitonic sort of n2 (power of two) keys in shared memory,
// ascending; returns after a block barrier.  Stages whose partners lie within
// one 64-key chunk (distance 32 or less) run warp by warp: warp w owns the
// chunks w, w + warps, ... and syncs only itself, so of the log2(n2) (log2(n2)
// + 1) / 2 stages only those of distance 64 or more wait for the whole block
// (15 of 66 for 2048 keys).  blockDim.x is a multiple of 32.
static __device__ void bitonic_sort(Key128 *keys, int n2)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarp = blockDim.x >> 5;
    const int nch = n2 >> 6;  // 64-key chunks
    if (nch == 0) {  // fewer than 64 keys: every stage block-wide
        for (int k = 2; k <= n2; k <<= 1)
            for (int j = k >> 1; j > 0; j >>= 1) {
                for (int i = threadIdx.x; i < n2; i += blockDim.x)
                    if ((i & j) == 0)
                        bitonic_cmpx(keys, i, k, j);
                __syncthreads();
            }
        __syncthreads();
        return;
    }
    // blocks of up to 64 keys: each chunk sorted by its warp, alternately
    // ascending and descending (the direction bit k of the key index)
    for (int c = warp; c < nch; c += nwarp)
        for (int k = 2; k <= 64; k <<= 1)
            for (int j = k >> 1; j > 0; j >>= 1) {
                bitonic_cmpx(keys, bitonic_pair(c, lane, j), k, j);
                __syncwarp();
            }
    __syncthreads();
    for (int k = 128; k <= n2; k <<= 1) {
        for (int j = k >> 1; j >= 64; j >>= 1) {
            for (int i = threadIdx.x; i < n2; i += blockDim.x)
                if ((i & j) == 0)
                    bitonic_cmpx(keys, i, k, j);
            __syncthreads();
        }
        for (int c = warp; c < nch; c += nwarp)
            for (int j = 32; j > 0; j >>= 1) {
                bitonic_cmpx(keys, bitonic_pair(c, lane, j), k, j);
                __syncwarp();
            }
        __syncthreads();
    }
}

__device__ __forceinline__ uint32_t cum_desc_key(int32_t cum)
{
    return 0xffffffffu - ((uint32_t)cum ^ 0x80000000u);  // larger cum -> smaller key
}

__device__ __forceinline__ int lower_bound_u64(const uint64_t *a, int n, uint64_t x)
{
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (a[mid] < x)
            lo = mid + 1;
        else
            hi = mid;
    }
    return lo;
}

template <typename CellT>
__global__ void __launch_bounds__(kThreads)
select_kernel(DevConfig cf, int cap, int parity, int F, const int32_t *__restrict__ n_parent,
              const int32_t *__restrict__ parent_cum, const uint8_t *__restrict__ parent_live,
              const CellT *__restrict__ cand_grids, const int32_t *__restrict__ cand_reward,
              const uint8_t *__restrict__ cand_done, const uint64_t *__restrict__ cand_hash, int k,
              CellT *next_grids, int32_t *next_cum, uint64_t *next_hash, uint8_t *next_live,
              int32_t *n_next, uint64_t *visited, int32_t *n_visited, uint32_t *status)
{
    extern __shared__ __align__(16) unsigned char smem[];
    Key128 *keys = reinterpret_cast<Key128 *>(smem);
    __shared__ int s_count;
    const int b = blockIdx.x, tid = threadIdx.x, HW = cf.HW;
    const int nc = 5 * F;
    int n2 = 1;
    while (n2 < nc)
        n2 <<= 1;
    const uint64_t *vis_in = visited + ((size_t)parity * cf.B + b) * cap;
    uint64_t *vis_out = visited + ((size_t)(parity ^ 1) * cf.B + b) * cap;
    const int nv = n_visited[b];
    const int np = n_parent[b];
    if (nv < 0 || nv > cap) {
        // a count the set cannot hold (block-uniform): nothing of the set is
        // read as hashes; the env selects nothing and keeps its set as given
        if (tid == 0) {
            atomicOr(status, kStatusVisitedCount);
            n_next[b] = 0;
        }
        for (int s = tid; s < k; s += blockDim.x) {
            next_cum[(size_t)b * k + s] = 0;
            next_hash[(size_t)b * k + s] = 0;
            next_live[(size_t)b * k + s] = 0;
        }
        for (int i = tid; i < cap; i += blockDim.x)
            vis_out[i] = vis_in[i];
        return;
    }

    // 1. candidates that exist and are not yet visited; key (hash, cum desc, index)
    for (int i = tid; i < n2; i += blockDim.x) {
        Key128 key = {~0ull, ~0ull};
        if (i < nc) {
            const int f = i / 5;
            const size_t gi = (size_t)b * F + f;
            if (f < np && parent_live[gi]) {
                const uint64_t hsh = cand_hash[(size_t)b * nc + i];
                const int pos = lower_bound_u64(vis_in, nv, hsh);
                if (pos == nv || vis_in[pos] != hsh) {
                    const int32_t cum = parent_cum[gi] + cand_reward[(size_t)b * nc + i];
                    key.hi = hsh;
                    key.lo = ((uint64_t)cum_desc_key(cum) << 32) | (uint32_t)i;
                }
            }
        }
        keys[i] = key;
    }
    __syncthreads();
    bitonic_sort(keys, n2);

    // 2. keep the first of each equal-hash run (highest cum, then lowest index);
    //    re-key as (cum desc, hash, index) for ranking.  Sentinels stay last.
    Key128 mine[kMaxCand / kThreads];
    int nm = 0;
    for (int i = tid; i < n2; i += blockDim.x) {
        const Key128 x = keys[i];
        Key128 r = {~0ull, ~0ull};
        const bool real = !(x.hi == ~0ull && x.lo == ~0ull);
        if (real && (i == 0 || keys[i - 1].hi != x.hi)) {
            r.hi = ((x.lo >> 32) << 32) | (x.hi >> 32);
            r.lo = (x.hi << 32) | (x.lo & 0xffffffffull);
        }
        mine[nm++] = r;
    }
    __syncthreads();
    nm = 0;
    for (int i = tid; i < n2; i += blockDim.x)
        keys[i] = mine[nm++];
    if (tid == 0)
        s_count = 0;
    __syncthreads();
    int cnt = 0;
    for (int i = tid; i < n2; i += blockDim.x)
        cnt += !(keys[i].hi == ~0ull && keys[i].lo == ~0ull);
    cnt = __reduce_add_sync(0xffffffffu, cnt);
    if ((tid & 31) == 0 && cnt)
        atomicAdd(&s_count, cnt);
    bitonic_sort(keys, n2);  // also orders s_count's writes before the read below
    const int take = min(k, s_count);

    // 3. next frontier
    for (int s = tid; s < take; s += blockDim.x) {
        const Key128 x = keys[s];
        const int idx = (int)(x.lo & 0xffffffffull);
        const uint64_t hsh = (x.hi << 32) | (x.lo >> 32);
        const int f = idx / 5;
        const size_t gi = (size_t)b * F + f;
        next_cum[(size_t)b * k + s] = parent_cum[gi] + cand_reward[(size_t)b * nc + idx];
        next_hash[(size_t)b * k + s] = hsh;
        next_live[(size_t)b * k + s] = (uint8_t)!cand_done[(size_t)b * nc + idx];
    }
    for (int s = take + tid; s < k; s += blockDim.x) {
        next_cum[(size_t)b * k + s] = 0;
        next_hash[(size_t)b * k + s] = 0;
        next_live[(size_t)b * k + s] = 0;
    }
    for (int e = tid; e < take * HW; e += blockDim.x) {
        const int s = e / HW, p = e - s * HW;
        const int idx = (int)(keys[s].lo & 0xffffffffull);
        next_grids[((size_t)b * k + s) * HW + p] = cand_grids[((size_t)b * nc + idx) * HW + p];
    }
    if (tid == 0)
        n_next[b] = take;

    // 4. visited := merge(visited, selected hashes), into the other buffer
    __syncthreads();
    uint64_t *sel = reinterpret_cast<uint64_t *>(keys + n2);  // sorted selected hashes
    int t2 = 1;
    while (t2 < take)
        t2 <<= 1;
    Key128 *hk = keys + n2 + (n2 + 1) / 2;  // scratch after sel (n2 uint64 = n2/2 Key128)
    for (int i = tid; i < t2; i += blockDim.x) {
        Key128 z = {~0ull, ~0ull};
        if (i < take)
            z = Key128{(keys[i].hi << 32) | (keys[i].lo >> 32), 0ull};
        hk[i] = z;
    }
    __syncthreads();
    bitonic_sort(hk, t2);
    for (int i = tid; i < take; i += blockDim.x)
        sel[i] = hk[i].hi;
    __syncthreads();
    if (nv + take > cap) {
        if (tid == 0) {
            atomicOr(status, kStatusVisitedOverflow);
            n_visited[b] = nv;
        }
        for (int i = tid; i < cap; i += blockDim.x)  // the set as given, unused tail included
            vis_out[i] = vis_in[i];
        return;
    }
    for (int i = tid; i < nv; i += blockDim.x)
        vis_out[i + lower_bound_u64(sel, take, vis_in[i])] = vis_in[i];
    for (int j = tid; j < take; j += blockDim.x)
        vis_out[j + lower_bound_u64(vis_in, nv, sel[j])] = sel[j];
    for (int i = nv + take + tid; i < cap; i += blockDim.x)  // the unused tail as given
        vis_out[i] = vis_in[i];
    if (tid == 0)
        n_visited[b] = nv + take;
}

// ------------------------------------------------- selection with hash tables
// av_select on a handle.  The visited states of env b live in an
// open-addressing table vtab[b][0, T) of 64-bit hashes (T a power of two with
// T >= 2 x capacity, so it is at most half full and every probe sequence ends
// at an empty slot); 0 marks an empty slot and vzero[b] records the state
// whose hash is 0.  A probe starts at mix64(hash) mod T and walks forward.
// One CTA per env:
//   1. each candidate that exists and is not visited goes into a shared-memory
//      table keyed by hash, keeping per hash the smallest (cum desc, index),
//      i.e. the highest cumulative reward and then the lowest index;
//   2. the distinct candidates are compacted and sorted once by (cum desc,
//      hash asc); the first k form the next frontier;
//   3. their hashes are added to the visited table (all are new: step 1 kept
//      only states not visited, one per hash).
// The result is the selection the sorted-array kernel (select_kernel) makes.

__device__ __forceinline__ uint32_t vis_slot(uint64_t h, uint32_t mask) { return (uint32_t)mix64(h) & mask; }

__device__ __forceinline__ bool vis_contains(const uint64_t *tab, uint32_t mask, uint32_t zero, uint64_t h)
{
    if (h == 0)
        return zero != 0u;
    uint32_t slot = vis_slot(h, mask);
    for (uint32_t probe = 0; probe <= mask; ++probe) {
        const uint64_t v = tab[slot];
        if (v == h)
            return true;
        if (v == 0)
            return false;
        slot = (slot + 1) & mask;
    }
    return false;
}

// Insert h (not present, nonzero) into a table with a free slot.
__device__ __forceinline__ void vis_insert(uint64_t *tab, uint32_t mask, uint64_t h)
{
    uint32_t slot = vis_slot(h, mask);
    for (uint32_t probe = 0; probe <= mask; ++probe) {
        const unsigned long long prev =
            atomicCAS(reinterpret_cast<unsigned long long *>(tab + slot), 0ull, (unsigned long long)h);
        if (prev == 0ull || prev == (unsigned long long)h)
            return;
        slot = (slot + 1) & mask;
    }
}

template <typename CellT>
__global__ void __launch_bounds__(kThreads)
search_init_hash_kernel(DevConfig cf, uint32_t vmask, const CellT *__restrict__ roots, uint64_t *root_hash,
                        uint8_t *root_live, uint64_t *vtab, uint32_t *vzero, int32_t *n_visited)
{
    // one thread per env; the tables were cleared before the launch
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= cf.B)
        return;
    const CellT *g = roots + (size_t)b * cf.HW;
    const uint32_t tiles = (1u << cf.C) - 1u;
    uint64_t hsh = 0xcbf29ce484222325ULL;
    int goal = cf.ch_goal < 0;
    for (int p = 0; p < cf.HW; ++p) {
        const uint32_t v = (uint32_t)g[p] & tiles;
        hsh = (hsh ^ (v & 0xffu)) * 0x100000001b3ULL;
        if (sizeof(CellT) == 2)
            hsh = (hsh ^ (v >> 8)) * 0x100000001b3ULL;
        if (cf.ch_goal >= 0)
            goal |= (int)((v >> cf.ch_goal) & 1u);
    }
    root_hash[b] = hsh;
    root_live[b] = (uint8_t)goal;
    if (hsh == 0)
        vzero[b] = 1u;
    else
        vis_insert(vtab + (size_t)b * (vmask + 1), vmask, hsh);
    n_visited[b] = 1;
}

// Shared memory of select_hash_kernel for 5 * F candidates.
__host__ __device__ inline uint32_t select_hash_slots(int F)
{
    uint32_t t = 64;
    while (t < 2u * 5u * (uint32_t)F)
        t <<= 1;
    return t;
}
inline size_t select_hash_smem_bytes(int F)
{
    int n2 = 1;
    while (n2 < 5 * F)
        n2 <<= 1;
    return (size_t)select_hash_slots(F) * 16 + (size_t)n2 * sizeof(Key128) + 64;
}

constexpr int kSelectThreads = 1024;  // threads of select_hash_kernel (one CTA per env)

template <typename CellT>
__global__ void __launch_bounds__(kSelectThreads)
select_hash_kernel(DevConfig cf, int cap, uint32_t vmask, int F, const int32_t *__restrict__ n_parent,
                   const int32_t *__restrict__ parent_cum, const uint8_t *__restrict__ parent_live,
                   const CellT *__restrict__ cand_grids, const int32_t *__restrict__ cand_reward,
                   const uint8_t *__restrict__ cand_done, const uint64_t *__restrict__ cand_hash, int k,
                   CellT *next_grids, int32_t *next_cum, uint64_t *next_hash, uint8_t *next_live,
                   int32_t *n_next, uint64_t *vtab, uint32_t *vzero, int32_t *n_visited, uint32_t *status)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const uint32_t T = select_hash_slots(F), smask = T - 1;
    unsigned long long *skey = reinterpret_cast<unsigned long long *>(smem);
    unsigned long long *sval = skey + T;
    Key128 *keys = reinterpret_cast<Key128 *>(sval + T);
    __shared__ unsigned long long s_zero_val;
    __shared__ int s_count;
    const int b = blockIdx.x, tid = threadIdx.x, HW = cf.HW;
    const int nc = 5 * F;
    const uint64_t *vt = vtab + (size_t)b * (vmask + 1);
    const uint32_t vz = vzero[b];
    const int np = n_parent[b];

    for (uint32_t i = tid; i < T; i += blockDim.x) {
        skey[i] = 0ull;
        sval[i] = ~0ull;
    }
    if (tid == 0) {
        s_zero_val = ~0ull;
        s_count = 0;
    }
    __syncthreads();

    // 1. candidates that exist and are not yet visited, one per hash
    for (int i = tid; i < nc; i += blockDim.x) {
        const int f = i / 5;
        const size_t gi = (size_t)b * F + f;
        if (f >= np || !parent_live[gi])
            continue;
        const uint64_t hsh = cand_hash[(size_t)b * nc + i];
        if (vis_contains(vt, vmask, vz, hsh))
            continue;
        const int32_t cum = parent_cum[gi] + cand_reward[(size_t)b * nc + i];
        const unsigned long long packed = ((unsigned long long)cum_desc_key(cum) << 32) | (uint32_t)i;
        if (hsh == 0) {
            atomicMin(&s_zero_val, packed);
            continue;
        }
        uint32_t slot = vis_slot(hsh, smask);
        for (uint32_t probe = 0; probe <= smask; ++probe) {
            const unsigned long long prev = atomicCAS(&skey[slot], 0ull, (unsigned long long)hsh);
            if (prev == 0ull || prev == (unsigned long long)hsh) {
                atomicMin(&sval[slot], packed);
                break;
            }
            slot = (slot + 1) & smask;
        }
    }
    __syncthreads();

    // 2. distinct candidates keyed (cum desc, hash, index), packed by warps
    //    (their order before the sort does not matter: the keys are distinct)
    const int lane = tid & 31;
    for (uint32_t i0 = tid & ~31u; i0 <= T; i0 += blockDim.x) {
        const uint32_t i = i0 + lane;
        uint64_t hsh = 0ull;
        unsigned long long v = ~0ull;
        bool have = false;
        if (i < T) {
            hsh = skey[i];
            v = sval[i];
            have = hsh != 0ull;
        } else if (i == T) {
            v = s_zero_val;
            have = v != ~0ull;
        }
        const uint32_t m = __ballot_sync(0xffffffffu, have);
        int base = 0;
        if (lane == 0 && m)
            base = atomicAdd(&s_count, __popc(m));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (have) {
            const int pos = base + __popc(m & ((1u << lane) - 1u));
            keys[pos].hi = ((v >> 32) << 32) | (hsh >> 32);
            keys[pos].lo = (hsh << 32) | (v & 0xffffffffull);
        }
    }
    __syncthreads();
    const int nu = s_count;
    int n2 = 1;
    while (n2 < nu)
        n2 <<= 1;
    for (int i = nu + tid; i < n2; i += blockDim.x)
        keys[i] = Key128{~0ull, ~0ull};
    __syncthreads();
    bitonic_sort(keys, n2);
    const int take = min(k, nu);

    // 3. next frontier
    for (int s = tid; s < take; s += blockDim.x) {
        const Key128 x = keys[s];
        const int idx = (int)(x.lo & 0xffffffffull);
        const uint64_t hsh = (x.hi << 32) | (x.lo >> 32);
        const size_t gi = (size_t)b * F + idx / 5;
        next_cum[(size_t)b * k + s] = parent_cum[gi] + cand_reward[(size_t)b * nc + idx];
        next_hash[(size_t)b * k + s] = hsh;
        next_live[(size_t)b * k + s] = (uint8_t)!cand_done[(size_t)b * nc + idx];
    }
    for (int s = take + tid; s < k; s += blockDim.x) {
        next_cum[(size_t)b * k + s] = 0;
        next_hash[(size_t)b * k + s] = 0;
        next_live[(size_t)b * k + s] = 0;
    }
    const size_t board = (size_t)HW * sizeof(CellT);
    if (board % 16 == 0 && (reinterpret_cast<uintptr_t>(cand_grids) & 15u) == 0 &&
        (reinterpret_cast<uintptr_t>(next_grids) & 15u) == 0) {
        const int n16 = (int)(board / 16);  // 16-byte pieces per board
        const uint4 *src = reinterpret_cast<const uint4 *>(cand_grids);
        uint4 *dst = reinterpret_cast<uint4 *>(next_grids);
        for (int e = tid; e < take * n16; e += blockDim.x) {
            const int s = e / n16, p = e - s * n16;
            const int idx = (int)(keys[s].lo & 0xffffffffull);
            dst[((size_t)b * k + s) * n16 + p] = src[((size_t)b * nc + idx) * n16 + p];
        }
    } else {
        for (int e = tid; e < take * HW; e += blockDim.x) {
            const int s = e / HW, p = e - s * HW;
            const int idx = (int)(keys[s].lo & 0xffffffffull);
            next_grids[((size_t)b * k + s) * HW + p] = cand_grids[((size_t)b * nc + idx) * HW + p];
        }
    }
    if (tid == 0)
        n_next[b] = take;

    // 4. the selected states join the visited set
    const int nv = n_visited[b];
    if (nv + take > cap) {
        if (tid == 0)
            atomicOr(status, kStatusVisitedOverflow);
        return;  // the set stays as it was, as with the sorted arrays
    }
    uint64_t *vw = vtab + (size_t)b * (vmask + 1);
    for (int s = tid; s < take; s += blockDim.x) {
        const uint64_t hsh = (keys[s].hi << 32) | (keys[s].lo >> 32);
        if (hsh == 0)
            vzero[b] = 1u;
        else
            vis_insert(vw, vmask, hsh);
    }
    if (tid == 0)
        n_visited[b] = nv + take;
}

// ------------------------------------------------------------ host helpers
inline size_t select_smem_bytes(int F)
{
    int n2 = 1;
    while (n2 < 5 * F)
        n2 <<= 1;
    // sort keys (n2) + selected hashes (n2 uint64) + their sort keys (n2)
    return (size_t)n2 * sizeof(Key128) * 2 + (size_t)n2 * 8 + 64;
}

// Anchor words per lane: the smallest power of two with 8 * NA >= NW.
inline int anchor_slots(int NW)
{
    int na = 1;
    while (8 * na < NW)
        na <<= 1;
    return na;
}

// Paths: cf.path 0 = choose, 1 = block per env, 2 = fast rollout (several warps
// per env), 3 = one warp per env, 4 = the memoising rollout.
// Rollouts: the memoising rollout (k_memo_impl.cuh) for boards of at most 16
// plane words, any rule count; else (or when forced) the block kernel.  The
// one-warp kernel (at most 16 rules) and the fast kernel (at most 64 rules)
// run when AV_KERNEL_PATH asks for them.  Expansion: one warp per parent for
// boards of at most 16 plane words unless the block path is forced.
inline bool use_memo_rollout(const DevConfig &cf) { return cf.NA <= 2 && (cf.path == 0 || cf.path == 4); }
inline bool use_env_warp_rollout(const DevConfig &cf) { return cf.NA <= 2 && cf.R <= 16 && cf.path == 3; }
inline bool use_fast_rollout(const DevConfig &cf)
{
    return cf.NA <= 2 && cf.R <= 64 && (cf.path == 2 || cf.path == 3);
}
// Variant semantics: one warp per environment for small boards with at most
// 16 rules unless the rule set is flagged busy or another path is forced.
inline bool use_variant_warp(const DevConfig &cf)
{
    return cf.NA <= 2 && cf.R <= 16 && ((cf.path == 0 && !cf.busy) || cf.path == 3 || cf.path == 4);
}
inline bool use_warp_expand(const DevConfig &cf) { return cf.NA <= 2 && cf.path != 1; }

constexpr int kDynSmemLimit = 200 * 1024;

// Environments per CTA of the one-warp-per-environment rollout: four, fewer
// when their shared memory would not fit.
inline int env_warps_per_cta(const DevConfig &cf)
{
    int epb = 4;
    while (epb > 1 && (size_t)epb * fast_layout(cf).total > (size_t)kDynSmemLimit)
        epb /= 2;
    return epb;
}

}  // namespace av
