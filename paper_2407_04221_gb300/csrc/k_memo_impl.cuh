// k_memo_impl.cuh -- fused rollout that remembers, for the board in hand, the
// outcome of each action it has taken on it; included by k_memo_u8.cu and
// k_memo_u16.cu (boards of at most 16 plane words, any rule count).
//
// A step's result is a function of the board, the action and the step
// counter (Sec. 2.1: the rules are matched on the current board; the action
// enters only as the force tiles next to the player).  While a board stays
// unchanged, the step with action a always pays the same reward, writes the
// same SET / CLEAR bits and leaves the same goal count.  One CTA runs one
// environment and keeps, per action, the outcome of that step on the current
// board once it has been computed: its reward and whether a goal tile is left
// (an action whose step changes the board changes it at once, so the actions
// remembered are the ones that leave it as it is).  A launch walks its steps
// 32 at a time, one step per lane: every lane looks up its step's action, and
// the first step whose action has no outcome yet, or that triggers an
// auto-reset, ends the run of steps that merely repeat the board.  Those steps
// write their rewards, done flags and observations (the board's canonical
// bytes, held in registers) at once, the CTA's warps taking turns.  The step
// that ended the run is evaluated by all warps together (every rule on the
// board with that action's force, as the step-by-step kernels do, the rules
// shared out among the warps); if it leaves the board unchanged its outcome is
// remembered and the walk goes on, else its flips are applied (or the initial
// map restored) and everything remembered is dropped.  No outcome is guessed:
// each is computed once per board and action, so results are exactly those of
// the step-by-step kernels.  Every warp runs the same walk on the same data
// (the action draws, the remembered outcomes and the step counter are the same
// in each), so all of them reach each block barrier together.
#pragma once

#include <algorithm>

#include "launch.h"

namespace av {

constexpr int kMemoLead = 4;  // leading terms of each rule tested for all rules at once

// Shared memory of one environment (one CTA): the valid-anchor and column
// masks; tile planes 0..C-1, the force of the action being evaluated (plane
// C) and an all-zero plane C+1 (padding terms read it as absent and pass),
// doubled; per warp a SET and a CLEAR plane set (each warp ORs the outputs of
// its own rules there); for each of two board slots (the current board and
// the one before it) the flip planes of each action's step, the board's planes
// (flat) and its canonical bytes; the initial map's planes (flat); per rule its
// two header words (uint4 each) and its first kMemoLead terms in each rotation;
// per-warp reductions; the whole rule table when staged.
struct MemoLayout {
    size_t vm, masks, planes, acc, flip, bplanes, basep, hdr, lead, leadm, cells, red, rules, total;
};

// Warps per environment (CTA): AV_MEMO_WARPS=1|2|4|8, read by av_create, else 4.
__host__ __device__ inline int memo_warps(const DevConfig &cf)
{
    return cf.memo_warps == 1 || cf.memo_warps == 2 || cf.memo_warps == 8 ? cf.memo_warps : 4;
}

__host__ __device__ inline MemoLayout memo_layout(const DevConfig &cf, bool staged)
{
    MemoLayout L;
    const size_t pw = (size_t)cf.C * cf.NW * 4;  // one plane set, bytes
    L.vm = 0;
    L.masks = align16((size_t)kShapes * cf.NW * 4);
    L.planes = align16(L.masks + (size_t)3 * cf.NW * 4);
    L.acc = align16(L.planes + (size_t)(cf.C + 2) * cf.NWP * 8);
    L.flip = align16(L.acc + 2 * (size_t)memo_warps(cf) * pw);
    L.bplanes = align16(L.flip + 10 * pw);
    L.basep = align16(L.bplanes + 2 * pw);
    L.hdr = align16(L.basep + pw);
    L.lead = align16(L.hdr + (size_t)cf.R * 32);
    L.leadm = align16(L.lead + (size_t)cf.R * 4 * kMemoLead * 8);
    L.cells = align16(L.leadm + (size_t)cf.R * 32 * cf.NA * 4);
    L.red = align16(L.cells + 2 * align16((size_t)cf.HW * cf.cell_bytes));
    L.rules = align16(L.red + 64 * 4);
    L.total = align16(L.rules + (staged ? (size_t)cf.rule_words * 4 : 0));
    return L;
}

// Whether the whole rule table is copied into shared memory: when the
// environment's region with it still lets six environments share an SM (the
// register budget allows seven); else the table is read through the L1 cache,
// and only for rules that pass their leading terms.  On the trajectory
// workload (the largest table 31 KB with its region: seven per SM) staging
// took the launch from 18.3 to 16.1 ms.  AV_MEMO_STAGE=1 (copy) or 0 (do not),
// read by av_create, forces the choice for measurements.
inline bool memo_staged(const DevConfig &cf)
{
    if (cf.rule_words <= 0 || cf.memo_stage == 2)
        return false;
    const size_t total = memo_layout(cf, true).total;
    if (cf.memo_stage == 1)
        return total <= (size_t)kDynSmemLimit;
    return total * (size_t)std::max(1, 24 / memo_warps(cf)) <= (size_t)227 * 1024;
}

// This lane's share of a board's canonical bytes to dst (global): 16-byte
// stores (mode 0: the board size and dst 16-byte aligned), 4-byte stores
// (mode 1) or single bytes (mode 2); nothing at or past nbytes.
template <int NV>
__device__ __forceinline__ void memo_store(unsigned char *dst, const uint32_t (&v)[4 * NV], int nbytes, int mode)
{
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < NV; ++j) {
        const int off = 16 * (lane + 32 * j);
        if (off >= nbytes)
            continue;
        if (mode == 0) {
            *reinterpret_cast<uint4 *>(dst + off) = make_uint4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int o = off + 4 * i;
                if (mode == 1) {
                    if (o < nbytes)
                        *reinterpret_cast<uint32_t *>(dst + o) = v[4 * j + i];
                } else {
                    for (int k = 0; k < 4 && o + k < nbytes; ++k)
                        dst[o + k] = (unsigned char)(v[4 * j + i] >> (8 * k));
                }
            }
        }
    }
}

__host__ __device__ inline int memo_store_mode(const void *p, int nbytes)
{
    const uintptr_t a = reinterpret_cast<uintptr_t>(p);
    if (nbytes % 16 == 0 && a % 16 == 0)
        return 0;
    if (nbytes % 4 == 0 && a % 4 == 0)
        return 1;
    return 2;
}

// Shared memory of one environment, as pointers.
struct MemoSmem {
    uint2 *planes;
    uint32_t *acc;   // [warp][SET, CLEAR][C * NW]
    uint32_t *flip;     // [slot][action][C * NW]: the bits each remembered step flips
    uint32_t *bplanes;  // [slot][C * NW]: each slot's board
    uint32_t *basep, *vm, *masks, *cells;
    int *red;  // two sets of 32 (alternate evaluations): [w] the reward of warp w's rules,
               // [8 + w] warp w's flags (bit 0: a bit flips, bit 1: a goal tile is left),
               // [16], [17] rules 0-31 / 32-63 that pass their leading terms
    const uint4 *hdr;   // [R][2]: (n_present, n_absent, n_out, reward), (first term, first output, shapes, 0)
    const uint2 *lead;  // [R][4 rotations][kMemoLead] term descriptors
    uint32_t *leadm;    // [R][32 lanes][NA]: the anchors that pass each rule's leading terms
};

// Anchors of this lane's words at which the first kMemoLead terms of rules r0,
// r0 + step, ... (KB of them) pass: the valid-anchor mask of the lane's
// rotation ANDed with each term's shifted plane word, absent terms
// complemented.  All loads are issued before any test, so the warp has
// independent work while it waits; rules past the table's end give no anchors.
template <int NA, int KB>
__device__ __forceinline__ void memo_lead_batch(const DevConfig &cf, const MemoSmem &S, uint32_t pbase, int r0,
                                                int step, uint32_t (&m)[KB][NA])
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    uint32_t shapes[KB];
    uint4 d01[KB], d23[KB];
    bool ok[KB];
#pragma unroll
    for (int k = 0; k < KB; ++k) {
        ok[k] = r0 + k * step < cf.R;
        const int r = ok[k] ? r0 + k * step : r0;
        shapes[k] = S.hdr[2 * r + 1].z;
        d01[k] = *reinterpret_cast<const uint4 *>(S.lead + (r * 4 + g) * kMemoLead);
        d23[k] = *reinterpret_cast<const uint4 *>(S.lead + (r * 4 + g) * kMemoLead + 2);
    }
#pragma unroll
    for (int k = 0; k < KB; ++k) {
        const uint32_t *vmr = S.vm + ((shapes[k] >> (8 * g)) & 0xffu) * cf.NW;
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            const int a = q + 8 * u;
            m[k][u] = ok[k] && a < cf.NW ? vmr[a] : 0u;
        }
    }
#pragma unroll
    for (int k = 0; k < KB; ++k) {
        const uint32_t dx[4] = {d01[k].x, d01[k].z, d23[k].x, d23[k].z};
        const uint32_t dy[4] = {d01[k].y, d01[k].w, d23[k].y, d23[k].w};
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            uint32_t x = m[k][u];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const uint2 w = lds2(pbase + dx[j] + 64 * u);
                x &= __funnelshift_r(w.x, w.y, dy[j]) ^ (uint32_t)((int32_t)dy[j] >> 31);
            }
            m[k][u] = x;
        }
    }
}

// The outputs of one rule (n_out entries at `op`, this lane's rotation) at
// the live anchors m of its four rotations, ORed into this warp's SET / CLEAR
// planes without atomics.  Output entry at window offset s = 32 d + sh moves
// the anchors of word j to word j + d (shifted left by sh) and j + d + 1; so
// the owner of word W takes (M[W - d] << sh) | (M[W - d - 1] >> (32 - sh)),
// fetching its rotation's match words by shuffles (word j of a rotation is lane
// (j & 7) of its quarter, anchor-word slot j >> 3).  The four rotations' words
// are ORed by two xor-shuffles, and the lanes of quarter 0 write each word
// (one lane per word, a plain read-modify-write in the warp's own planes).
template <int NA, bool SM>
__device__ __forceinline__ void memo_write(const DevConfig &cf, const uint4 *op, uint32_t n_out,
                                           const uint32_t (&m)[NA], uint32_t *wset, uint32_t *wclr)
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    for (uint32_t o = 0; o < n_out; ++o) {
        const uint4 ov = SM ? op[4 * o] : __ldg(op + 4 * o);
        const int d = (int)ov.x;
        const uint32_t sh = ov.y;
        uint32_t cw[NA];
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            const int a = q + 8 * u - d, b = a - 1;  // source words of the low and high parts
            uint32_t xa = 0, xb = 0;
#pragma unroll
            for (int v = 0; v < NA; ++v) {
                const uint32_t ya = __shfl_sync(0xffffffffu, m[v], (g << 3) | (a & 7));
                const uint32_t yb = __shfl_sync(0xffffffffu, m[v], (g << 3) | (b & 7));
                if (a >= 0 && (a >> 3) == v)
                    xa = ya;
                if (b >= 0 && (b >> 3) == v)
                    xb = yb;
            }
            uint32_t c = (xa << sh) | (sh ? (xb >> (32u - sh)) : 0u);
            c |= __shfl_xor_sync(0xffffffffu, c, 8);
            c |= __shfl_xor_sync(0xffffffffu, c, 16);
            cw[u] = c;
        }
        if (g == 0) {
#pragma unroll
            for (int u = 0; u < NA; ++u) {
                const int W = q + 8 * u;
                if (W >= cf.NW || !cw[u])
                    continue;
                for (uint32_t ch = ov.z; ch; ch &= ch - 1)
                    wset[(__ffs(ch) - 1) * cf.NW + W] |= cw[u];
                for (uint32_t ch = ov.w; ch; ch &= ch - 1)
                    wclr[(__ffs(ch) - 1) * cf.NW + W] |= cw[u];
            }
        }
        __syncwarp();
    }
}

// One step of the board in S.planes with action `a`, by all NWARP warps of the
// CTA: every rule in its four rotations as in the step-by-step kernels: the
// force plane of `a`, the leading terms of every rule (warp w takes rules w,
// w + NWARP, ...), then the rules that pass them dealt out among the warps
// afresh, so that a few live rules do not fall to one warp: their remaining
// terms (four per
// vote), the outputs of live matches ORed into the warp's own SET / CLEAR
// planes (memo_write); then the flip planes flip_out (SET bits on clear cells,
// CLEAR bits on set cells, over every warp's planes).  `n_terms` is the
// table's term count (its word 1).  Returns
// (reward, bit 0: the step changes the board, bit 1: a goal tile is left
// after it, always without a goal channel), the same in every thread.  Not
// inlined: it runs once per board and action.
template <int NA, bool SM, int NWARP>
static __device__ __forceinline__ int2 memo_step_eval(DevConfig cf, const uint32_t *tab, uint32_t n_terms, MemoSmem S,
                                                       int a, uint32_t *flip_out, int &parity)
{
    constexpr int T = 32 * NWARP;
    constexpr int KB = 3;  // rules per warp whose leading terms are tested together
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 3, q = lane & 7;
    const int NW = cf.NW, NWP = cf.NWP, cnw = cf.C * NW;
    // the reductions alternate between two sets, so that no barrier is needed
    // after their last read: the set written here was last read two
    // evaluations ago, before the barriers of the one in between
    int *red = S.red + 32 * parity;
    parity ^= 1;
    for (int i = tid; i < 2 * NWARP * cnw; i += T)
        S.acc[i] = 0u;
    if (tid < 2)
        red[16 + tid] = 0;
    if (warp == NWARP - 1)
        force_plane(cf, S.planes, S.masks, a);
    __syncthreads();
    const uint32_t pbase = (uint32_t)__cvta_generic_to_shared(S.planes) + q * 8;
    // this warp's rules whose leading terms pass somewhere
    uint32_t alive0 = 0, alive1 = 0;
    for (int r0 = warp; r0 < cf.R; r0 += KB * NWARP) {
        uint32_t m[KB][NA];
        memo_lead_batch<NA, KB>(cf, S, pbase, r0, NWARP, m);
#pragma unroll
        for (int k = 0; k < KB; ++k) {
            uint32_t any = 0;
#pragma unroll
            for (int u = 0; u < NA; ++u)
                any |= m[k][u];
            const int r = r0 + k * NWARP;
            if (r < cf.R) {
#pragma unroll
                for (int u = 0; u < NA; ++u)  // kept for the warp that takes the rule on
                    S.leadm[(r * 32 + lane) * NA + u] = m[k][u];
            }
            if (any) {  // (rules past the end have no anchors)
                if (r < 32)
                    alive0 |= 1u << r;
                else
                    alive1 |= 1u << (r - 32);
            }
        }
    }
    alive0 = __reduce_or_sync(0xffffffffu, alive0);
    alive1 = cf.R > 32 ? __reduce_or_sync(0xffffffffu, alive1) : 0u;
    if (NWARP > 1) {
        // the rules that passed, dealt out afresh: the k-th of them to warp k mod NWARP
        if (lane == 0) {
            if (alive0)
                atomicOr(reinterpret_cast<unsigned int *>(red) + 16, alive0);
            if (alive1)
                atomicOr(reinterpret_cast<unsigned int *>(red) + 17, alive1);
        }
        __syncthreads();
        const uint32_t all0 = (uint32_t)red[16], all1 = (uint32_t)red[17];
        alive0 = alive1 = 0;
        int k = 0;
        for (uint32_t x = all0; x; x &= x - 1, ++k)
            if (k % NWARP == warp)
                alive0 |= x & (0u - x);
        for (uint32_t x = all1; x; x &= x - 1, ++k)
            if (k % NWARP == warp)
                alive1 |= x & (0u - x);
    }
    const uint2 *terms = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R));
    const uint4 *outs = reinterpret_cast<const uint4 *>(tab + table_outs_word(cf.R, n_terms));
    const uint32_t pass_x = (uint32_t)(cf.C + 1) * NWP * 8;  // a term on the zero plane, read as absent
    int rew = 0;
    for (int k = 0; k < 2; ++k) {
        uint32_t alive = k ? alive1 : alive0;
        while (alive) {
            const int r = 32 * k + __ffs(alive) - 1;
            alive &= alive - 1;
            uint32_t m[NA];
#pragma unroll
            for (int u = 0; u < NA; ++u)  // written by the warp that tested the leading terms
                m[u] = S.leadm[(r * 32 + lane) * NA + u];
            const uint4 h0 = S.hdr[2 * r], h1 = S.hdr[2 * r + 1];
            const uint32_t nt = h0.x + h0.y;
            const uint2 *tp = terms + (size_t)h1.x * 4 + g;
            bool live = true;
            for (uint32_t t = kMemoLead; live && t < nt; t += 4) {
                uint2 d[4];
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    d[j] = t + j < nt ? ld2<SM>(tp + 4 * (t + j)) : make_uint2(pass_x, kTermAbsent);
                uint32_t any = 0;
#pragma unroll
                for (int u = 0; u < NA; ++u) {
                    uint32_t x = m[u];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const uint2 w = lds2(pbase + d[j].x + 64 * u);
                        x &= __funnelshift_r(w.x, w.y, d[j].y) ^ (uint32_t)((int32_t)d[j].y >> 31);
                    }
                    m[u] = x;
                    any |= x;
                }
                live = __any_sync(0xffffffffu, any != 0u);
            }
            if (!live)
                continue;
            uint32_t cnt = 0;
#pragma unroll
            for (int u = 0; u < NA; ++u)
                cnt += __popc(m[u]);
            if (__any_sync(0xffffffffu, cnt != 0u)) {  // the rule matched: it pays and writes
                rew += (int)h0.w * (int)cnt;
                memo_write<NA, SM>(cf, outs + (size_t)h1.y * 4 + g, h0.z, m, S.acc + (size_t)warp * 2 * cnw,
                                   S.acc + (size_t)warp * 2 * cnw + cnw);
            }
        }
    }
    rew = __reduce_add_sync(0xffffffffu, rew);
    if (lane == 0)
        red[warp] = rew;
    __syncthreads();  // every warp's SET / CLEAR bits and reward
    uint32_t any = 0, goal = 0;
    for (int i = tid, c = tid / NW, w = tid - (tid / NW) * NW; i < cnw; i += T, c += T / NW, w += T % NW) {
        if (w >= NW) {  // (c, w) of i = c * NW + w, stepped by T = (T / NW) * NW + T % NW
            w -= NW;
            ++c;
        }
        uint32_t st = 0, cl = 0;
#pragma unroll
        for (int k = 0; k < NWARP; ++k) {
            st |= S.acc[2 * k * cnw + i];
            cl |= S.acc[(2 * k + 1) * cnw + i];
        }
        const uint32_t d = S.planes[c * NWP + w].x;
        const uint32_t f = (d & cl) | (~d & st);  // a bit changes where a match asks for it
        flip_out[i] = f;
        any |= f;
        if (c == cf.ch_goal)
            goal |= d ^ f;
    }
    any = __any_sync(0xffffffffu, any != 0u);
    goal = __any_sync(0xffffffffu, goal != 0u);
    if (lane == 0)
        red[8 + warp] = (any ? 1 : 0) | (goal ? 2 : 0);
    __syncthreads();  // the flip planes and flags
    int total = 0, flags = 0;
#pragma unroll
    for (int w = 0; w < NWARP; ++w) {
        total += red[w];
        flags |= red[8 + w];
    }
    const int bits = (flags & 1) | ((cf.ch_goal < 0 || (flags & 2)) ? 2 : 0);
    return make_int2(total, bits);
}

// The board after its step (planes ^= flip), written also into `bpl` (the
// other slot's flat planes), in one pass (all warps); returns whether it
// differs from what `bpl` held (every thread).
template <int NWARP>
static __device__ __forceinline__ int memo_apply_switch(const DevConfig &cf, uint2 *planes, const uint32_t *flip,
                                                         uint32_t *bpl)
{
    constexpr int T = 32 * NWARP;
    const int NW = cf.NW, NWP = cf.NWP, cnw = cf.C * NW, tid = threadIdx.x;
    int diff = 0;
    for (int i = tid, c = tid / NW, w = tid - (tid / NW) * NW; i < cnw; i += T, c += T / NW, w += T % NW) {
        if (w >= NW) {
            w -= NW;
            ++c;
        }
        const uint32_t f = flip[i], x = planes[c * NWP + w].x ^ f;
        if (f)
            put_word(planes, NWP, c, w, x);
        diff |= bpl[i] != x;
        bpl[i] = x;
    }
    return __syncthreads_or(diff);
}

// Auto-reset: the initial map's planes back into the tile planes (all warps).
// Returns whether the board differed from the initial map (every thread).
template <int NWARP>
static __device__ __forceinline__ int memo_restore(DevConfig cf, uint2 *planes, const uint32_t *basep)
{
    const int NW = cf.NW, NWP = cf.NWP, cnw = cf.C * NW;
    int diff = 0;
    constexpr int T = 32 * NWARP;
    const int tid = threadIdx.x;
    for (int i = tid, c = tid / NW, w = tid - (tid / NW) * NW; i < cnw; i += T, c += T / NW, w += T % NW) {
        if (w >= NW) {
            w -= NW;
            ++c;
        }
        const uint32_t b = basep[i];
        if (planes[c * NWP + w].x != b) {
            diff = 1;
            put_word(planes, NWP, c, w, b);
        }
    }
    return __syncthreads_or(diff);
}

// The current tile planes (flat) into `bpl` (all warps); returns whether they
// differed from what `bpl` held (every thread).
template <int NWARP>
static __device__ __forceinline__ int memo_switch(const DevConfig &cf, const uint2 *planes, uint32_t *bpl)
{
    constexpr int T = 32 * NWARP;
    const int NW = cf.NW, NWP = cf.NWP, cnw = cf.C * NW, tid = threadIdx.x;
    int diff = 0;
    for (int i = tid, c = tid / NW, w = tid - (tid / NW) * NW; i < cnw; i += T, c += T / NW, w += T % NW) {
        if (w >= NW) {
            w -= NW;
            ++c;
        }
        const uint32_t x = planes[c * NWP + w].x;
        diff |= bpl[i] != x;
        bpl[i] = x;
    }
    return __syncthreads_or(diff);
}

// This lane's 16-byte units of a board's canonical bytes from `cells`.
template <int NV>
__device__ __forceinline__ void memo_load_cells(const uint32_t *cells, int n16, uint32_t (&v)[4 * NV])
{
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < NV; ++j) {
        const int u = lane + 32 * j;
        const uint4 x = u < n16 ? reinterpret_cast<const uint4 *>(cells)[u] : make_uint4(0u, 0u, 0u, 0u);
        v[4 * j] = x.x;
        v[4 * j + 1] = x.y;
        v[4 * j + 2] = x.z;
        v[4 * j + 3] = x.w;
    }
}

template <typename T>
__device__ __forceinline__ void swap_vals(T &a, T &b)
{
    const T t = a;
    a = b;
    b = t;
}

// The board's canonical bytes into `cells` (shared, a whole number of
// 16-byte units, zero past the board) from the doubled tile planes (all
// warps), then this lane's 16-byte units of them into v.
template <typename CellT, int NV, int NWARP>
__device__ __forceinline__ void memo_cells(const DevConfig &cf, const uint2 *planes, uint32_t *cells,
                                           uint32_t (&v)[4 * NV])
{
    constexpr int kPer = 4 / (int)sizeof(CellT);  // cells per word
    const int HW = cf.HW, NWP = cf.NWP;
    const int n16 = (HW * (int)sizeof(CellT) + 15) / 16;
    for (int k = threadIdx.x; k < 4 * n16; k += 32 * NWARP) {
        const int p0 = k * kPer;
        uint32_t x = 0;
        if (p0 < HW) {
            const int w = p0 >> 5, b = p0 & 31;  // a word's cells lie in one plane word
            for (int c = 0; c < cf.C; ++c) {
                const uint32_t y = planes[c * NWP + w].x >> b;
                const uint32_t s = sizeof(CellT) == 1 ? ((y & 0xfu) * 0x00204081u) & 0x01010101u
                                                      : ((y & 0x3u) * 0x00008001u) & 0x00010001u;
                x |= s << c;
            }
        }
        cells[k] = x;
    }
    __syncthreads();
    memo_load_cells<NV>(cells, n16, v);
}

// Fused rollout, one CTA of NWARP warps per environment; see the top of this
// file.  With `actions` non-null the action of every step is actions[env]
// (av_step, n_steps = 1); else step s draws draw(seed, 4, env, 0, s) mod 5.
// Four warps: 72 registers a thread (seven CTAs per SM, which shared memory
// allows on the trajectory workload anyway: 13.7 against 14.0 ms at 64).
template <typename CellT, int NA, bool SM, int NWARP>
__global__ void __launch_bounds__(32 * NWARP, NWARP == 4 ? 7 : 32 / NWARP)
rollout_memo_kernel(DevConfig cf, const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
                    const uint32_t *__restrict__ vm_g, const uint32_t *__restrict__ masks_g, CellT *cur,
                    const CellT *__restrict__ init, int32_t *tsteps, int n_steps, uint64_t seed,
                    const uint8_t *__restrict__ actions, CellT *obs_traj, int32_t *rew_traj,
                    uint8_t *done_traj, int32_t *rew_sum, uint32_t *status, const int32_t *__restrict__ order,
                    uint32_t *cost)
{
    constexpr int T = 32 * NWARP;
    extern __shared__ __align__(16) unsigned char smem[];
    const long long clock0 = clock64();
    const MemoLayout L = memo_layout(cf, SM);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int env = order ? order[blockIdx.x] : (int)blockIdx.x;
    const int C = cf.C, NW = cf.NW, NWP = cf.NWP, HW = cf.HW, cnw = C * NW;
    const int nbytes = HW * (int)sizeof(CellT);
    MemoSmem S;
    S.planes = reinterpret_cast<uint2 *>(smem + L.planes);
    S.acc = reinterpret_cast<uint32_t *>(smem + L.acc);
    S.flip = reinterpret_cast<uint32_t *>(smem + L.flip);
    S.bplanes = reinterpret_cast<uint32_t *>(smem + L.bplanes);
    S.basep = reinterpret_cast<uint32_t *>(smem + L.basep);
    S.vm = reinterpret_cast<uint32_t *>(smem + L.vm);
    S.masks = reinterpret_cast<uint32_t *>(smem + L.masks);
    S.cells = reinterpret_cast<uint32_t *>(smem + L.cells);
    S.red = reinterpret_cast<int *>(smem + L.red);
    uint4 *hdr = reinterpret_cast<uint4 *>(smem + L.hdr);
    uint2 *lead = reinterpret_cast<uint2 *>(smem + L.lead);
    S.hdr = hdr;
    S.lead = lead;
    S.leadm = reinterpret_cast<uint32_t *>(smem + L.leadm);
    const int table = cf.rules_per_env ? env : 0;
    const uint32_t *tab_g = arena + tab_off[table];
    const uint32_t *tab = SM ? reinterpret_cast<const uint32_t *>(smem + L.rules) : tab_g;

    // ---- stage
    for (int i = tid; i < kShapes * NW; i += T)
        S.vm[i] = __ldg(vm_g + i);
    for (int i = tid; i < 3 * NW; i += T)
        S.masks[i] = __ldg(masks_g + i);
    if (SM) {
        const uint32_t n = tab_off[table + 1] - tab_off[table];
        for (uint32_t i = tid; i < n / 4; i += T)
            reinterpret_cast<uint4 *>(smem + L.rules)[i] = __ldg(reinterpret_cast<const uint4 *>(tab_g) + i);
    }
    for (int i = tid; i < 2 * cf.R; i += T)  // rule headers: words 4 + 8r .. 4 + 8r + 7 of the table
        hdr[i] = __ldg(reinterpret_cast<const uint4 *>(tab_g + 4) + i);
    for (int i = tid; i < (C + 2) * NWP; i += T)
        S.planes[i] = make_uint2(0u, 0u);
    const uint32_t n_terms = __ldg(tab_g + 1);
    {
        const uint2 *terms = reinterpret_cast<const uint2 *>(tab_g + table_terms_word(cf.R));
        const uint2 pass = make_uint2((uint32_t)(C + 1) * NWP * 8, kTermAbsent);
        for (int i = tid; i < cf.R * 4 * kMemoLead; i += T) {  // [rule][rotation][term]
            const int r = i / (4 * kMemoLead), g = (i / kMemoLead) & 3, j = i & (kMemoLead - 1);
            const uint32_t nt = __ldg(tab_g + 4 + 8 * r) + __ldg(tab_g + 5 + 8 * r);
            const uint32_t first = __ldg(tab_g + 8 + 8 * r);
            lead[i] = (uint32_t)j < nt ? __ldg(terms + (size_t)(first + j) * 4 + g) : pass;
        }
    }
    __syncthreads();  // the zeroed planes
    {
        // the boards into planes: warp w takes the 32-cell groups w, w + NWARP, ...
        const CellT *src = cur + (size_t)env * HW, *isrc = init + (size_t)env * HW;
        for (int base = 32 * warp; base < HW; base += T) {
            const int p = base + lane;
            const uint32_t x = p < HW ? (uint32_t)src[p] : 0u;
            const uint32_t xi = p < HW ? (uint32_t)isrc[p] : 0u;
            const int w = base >> 5;
            for (int c = 0; c < C; ++c) {
                const uint32_t bits = __ballot_sync(0xffffffffu, (x >> c) & 1u);
                const uint32_t ibits = __ballot_sync(0xffffffffu, (xi >> c) & 1u);
                if (lane == 0) {
                    put_word(S.planes, NWP, c, w, bits);
                    S.basep[c * NW + w] = ibits;
                }
            }
        }
    }
    __syncthreads();

    uint32_t v[4 * NA];  // this lane's 16-byte units of the board's canonical bytes
    // Two board slots: the current board (slot cs) and the one before it.  Per
    // slot: the board's planes (flat, S.bplanes) and canonical bytes (S.cells),
    // and the outcomes remembered for it, in registers the same in every warp:
    // bit a of kq[s] when action a leaves the board unchanged, of kc[s] when it
    // changes it (its flip planes kept in S.flip[s][a]), of gm[s] when a goal
    // tile is left after it; lane a holds its reward in rw[s].
    const int n16 = (HW * (int)sizeof(CellT) + 15) / 16;  // 16-byte units of a board
    // the current slot and the other one (swapped when the board changes)
    uint32_t *cells_c = S.cells, *cells_o = S.cells + 4 * n16;
    uint32_t *bpl_c = S.bplanes, *bpl_o = S.bplanes + cnw;
    uint32_t *flip_c = S.flip, *flip_o = S.flip + 5 * cnw;
    uint32_t kq = 0u, kc = 0u, gm = 0u, okq = 0u, okc = 0u, ogm = 0u;
    int rw = 0, orw = 0, valid_other = 0;
    int parity = 0;  // which set of reduction slots the next evaluation uses
    memo_switch<NWARP>(cf, S.planes, bpl_c);
    memo_cells<CellT, NA, NWARP>(cf, S.planes, cells_c, v);
    int t = tsteps[env];
    int sum = 0, warn = 0;
    const int obs_mode = obs_traj ? memo_store_mode(obs_traj, nbytes) : 0;
    const size_t step_stride = (size_t)cf.B * nbytes;  // bytes from one step's boards to the next's
    unsigned char *const obs_env = obs_traj ? reinterpret_cast<unsigned char *>(obs_traj) + (size_t)env * nbytes
                                            : nullptr;

    for (int b0 = 0; b0 < n_steps; b0 += 32) {
        const int lim = min(32, n_steps - b0);
        const int a_l = lane < lim ? action_at(actions, seed, env, b0 + lane, &warn) : 0;
        int l0 = 0;
        while (l0 < lim) {
            // lane l takes step b0 + l as if no step of this run before it
            // changed the board, reset the environment or had no remembered
            // outcome that leaves the board as it is
            const bool act = lane >= l0 && lane < lim;
            const bool q_l = (kq >> a_l) & 1u;
            const int r_l = __shfl_sync(0xffffffffu, rw, a_l);
            const bool goal_l = (gm >> a_l) & 1u;
            const int t_l = t + (lane - l0) + 1;
            const bool done_l = !goal_l || (cf.max_steps > 0 && t_l >= cf.max_steps);
            const uint32_t ev = __ballot_sync(0xffffffffu, act && (!q_l || (done_l && cf.auto_reset)));
            const int e = ev ? __ffs(ev) - 1 : lim;  // the first step that is not a plain repeat
            if (warp == 0 && act && lane < e) {  // steps that repeat the board
                sum += r_l;
                if (rew_traj)
                    rew_traj[(size_t)(b0 + lane) * cf.B + env] = r_l;
                if (done_traj)
                    done_traj[(size_t)(b0 + lane) * cf.B + env] = (uint8_t)done_l;
            }
            if (obs_traj) {  // the warps take turns
                unsigned char *o = obs_env + (size_t)(b0 + l0 + warp) * step_stride;
                for (int l = l0 + warp; l < e; l += NWARP, o += NWARP * step_stride)
                    memo_store<NA>(o, v, nbytes, obs_mode);
            }
            t += e - l0;
            if (e >= lim)
                break;

            // ---- step b0 + e (every warp)
            const int a = __shfl_sync(0xffffffffu, a_l, e);
            const uint32_t bit = 1u << a;
            uint32_t *fl = flip_c + (size_t)a * cnw;  // flip planes of the current board and action a
            int r, goal_left;
            bool moves;  // the step's own outcome changes the board
            if (kq & bit) {  // a remembered step that ends in an auto-reset
                r = __shfl_sync(0xffffffffu, rw, a);
                goal_left = (gm & bit) != 0u;
                moves = false;
            } else if (kc & bit) {  // a remembered step that changes the board
                r = __shfl_sync(0xffffffffu, rw, a);
                goal_left = (gm & bit) != 0u;
                moves = true;
            } else {
                const int2 o = memo_step_eval<NA, SM, NWARP>(cf, tab, n_terms, S, a, fl, parity);
                r = o.x;
                goal_left = (o.y & 2) != 0;
                moves = (o.y & 1) != 0;
                if (lane == a)
                    rw = r;
                if (goal_left)
                    gm |= bit;
                if (!moves) {  // the board stays: remember the outcome, take the step again
                    kq |= bit;
                    l0 = e;
                    continue;
                }
                kc |= bit;
            }
            t += 1;
            const int done = !goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
            int changed, diff_other = -1;  // whether the new board differs from the other slot's
            if (done && cf.auto_reset) {
                changed = memo_restore<NWARP>(cf, S.planes, S.basep);
                t = 0;
            } else {  // (a board-changing outcome: `moves` holds)
                diff_other = memo_apply_switch<NWARP>(cf, S.planes, fl, bpl_o);
                changed = 1;
            }
            if (warp == 0 && lane == e) {
                sum += r;
                if (rew_traj)
                    rew_traj[(size_t)(b0 + e) * cf.B + env] = r;
                if (done_traj)
                    done_traj[(size_t)(b0 + e) * cf.B + env] = (uint8_t)done;
            }
            if (changed) {
                // the new board goes to the other slot, which becomes the
                // current one: if it held the same board, its remembered
                // outcomes hold; else they are dropped
                const int same =
                    !(diff_other >= 0 ? diff_other : memo_switch<NWARP>(cf, S.planes, bpl_o)) && valid_other;
                swap_vals(cells_c, cells_o);
                swap_vals(bpl_c, bpl_o);
                swap_vals(flip_c, flip_o);
                swap_vals(kq, okq);
                swap_vals(kc, okc);
                swap_vals(gm, ogm);
                swap_vals(rw, orw);
                if (same) {
                    memo_load_cells<NA>(cells_c, n16, v);
                } else {
                    kq = kc = gm = 0u;
                    memo_cells<CellT, NA, NWARP>(cf, S.planes, cells_c, v);
                }
                valid_other = 1;
            }
            if (obs_traj && warp == (e % NWARP))
                memo_store<NA>(obs_env + (size_t)(b0 + e) * step_stride, v, nbytes, obs_mode);
            l0 = e + 1;
        }
    }
    if (warp == 0) {
        memo_store<NA>(reinterpret_cast<unsigned char *>(cur) + (size_t)env * nbytes, v, nbytes,
                       memo_store_mode(cur, nbytes));
        sum = __reduce_add_sync(0xffffffffu, sum);
        warn = __any_sync(0xffffffffu, warn);
        if (lane == 0) {
            tsteps[env] = t;
            if (rew_sum)
                rew_sum[env] = sum;
            if (warn)
                atomicOr(status + 1, kWarnAction);
            if (cost)  // this launch's time for the environment, in units of 256 cycles
                cost[env] = (uint32_t)min((clock64() - clock0) >> 8, 0xffffffffLL);
        }
    }
}

#ifdef AV_MEMO_ORDER
// Launch order of the next memoising rollout (one CTA): environments by
// decreasing cost in the last launch, in power-of-two buckets (a counting
// sort; the order within a bucket is arbitrary).  Started first, the costly
// environments no longer finish after everything else.
__global__ void __launch_bounds__(1024) memo_order_kernel(const uint32_t *__restrict__ cost, int32_t *order, int B)
{
    __shared__ int hist[33], next[33];
    const int tid = threadIdx.x;
    if (tid < 33)
        hist[tid] = 0;
    __syncthreads();
    for (int i = tid; i < B; i += blockDim.x)
        atomicAdd(&hist[32 - __clz(cost[i])], 1);
    __syncthreads();
    if (tid == 0) {
        int s = 0;
        for (int b = 32; b >= 0; --b) {
            next[b] = s;
            s += hist[b];
        }
    }
    __syncthreads();
    for (int i = tid; i < B; i += blockDim.x)
        order[atomicAdd(&next[32 - __clz(cost[i])], 1)] = i;
}

void launch_memo_order(const uint32_t *cost, int32_t *order, int B, cudaStream_t st)
{
    memo_order_kernel<<<1, 1024, 0, st>>>(cost, order, B);
}
#endif

}  // namespace av

// ---------------------------------------------------------------- launchers
// Compiled once per cell type (AV_MEMO_CELL) by k_memo_u8.cu / k_memo_u16.cu.
#ifdef AV_MEMO_CELL
namespace av {
namespace AV_MEMO_NS {

template <typename CellT, int NA, bool SM, int NWARP>
void memo_t(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
            const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
            const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
            uint32_t *status, const int32_t *order, uint32_t *cost, cudaStream_t st)
{
    const size_t sm = memo_layout(cf, SM).total;
    rollout_memo_kernel<CellT, NA, SM, NWARP><<<cf.B, 32 * NWARP, sm, st>>>(
        cf, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
        (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status, order, cost);
}

template <typename CellT, int NA, bool SM>
void memo_w(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
            const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
            const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
            uint32_t *status, const int32_t *order, uint32_t *cost, cudaStream_t st)
{
#define AV_MEMO(NWARP)                                                                                     \
    memo_t<CellT, NA, SM, NWARP>(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj, \
                                 rew_traj, done_traj, rew_sum, status, order, cost, st)
    switch (memo_warps(cf)) {
    case 1: AV_MEMO(1); break;
    case 2: AV_MEMO(2); break;
    case 8: AV_MEMO(8); break;
    default: AV_MEMO(4); break;
    }
#undef AV_MEMO
}

}  // namespace AV_MEMO_NS

cudaError_t AV_MEMO_CONFIGURE()
{
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    };
#define AV_SETM(NA, SM) \
    set((const void *)rollout_memo_kernel<AV_MEMO_CELL, NA, SM, 1>); \
    set((const void *)rollout_memo_kernel<AV_MEMO_CELL, NA, SM, 2>); \
    set((const void *)rollout_memo_kernel<AV_MEMO_CELL, NA, SM, 4>); \
    set((const void *)rollout_memo_kernel<AV_MEMO_CELL, NA, SM, 8>);
    AV_SETM(1, true)
    AV_SETM(1, false)
    AV_SETM(2, true)
    AV_SETM(2, false)
#undef AV_SETM
    return e;
}

void AV_MEMO_LAUNCH(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
                    const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
                    const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj,
                    int32_t *rew_sum, uint32_t *status, const int32_t *order, uint32_t *cost, cudaStream_t st)
{
#define AV_MEMO(NA, SM)                                                                                  \
    AV_MEMO_NS::memo_w<AV_MEMO_CELL, NA, SM>(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed,   \
                                             actions, obs_traj, rew_traj, done_traj, rew_sum, status, order,  \
                                             cost, st)
    const bool staged = memo_staged(cf);
    if (cf.NA == 1) {
        if (staged) AV_MEMO(1, true);
        else AV_MEMO(1, false);
    } else {
        if (staged) AV_MEMO(2, true);
        else AV_MEMO(2, false);
    }
#undef AV_MEMO
}

}  // namespace av
#endif
