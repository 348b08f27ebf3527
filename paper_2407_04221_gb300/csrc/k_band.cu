// k_band.cu -- rollouts of boards larger than one CTA's shared memory (up to
// 256 x 256 cells): the same step (Sec. 2.1; match, write, combine) with the
// board streamed through shared memory in bands of rows.
//
// One CTA of kThreads per environment.  The board's bit-planes (C tile
// channels and the force plane, plain 32-bit words) and its SET / CLEAR
// accumulators live in global memory, where they stay in L2.  Each step
// visits the bands in turn: a band is `band_rows` rows of anchors plus the
// rows below it that windows anchored in it reach (four for 5 x 5 patterns),
// `band_nw` plane words in all.  The CTA copies the band's planes into shared
// memory in the doubled (word j, word j + 1) layout, derives the band's
// valid-anchor masks from the whole board's (anchors outside the band's rows
// cleared), runs the block rollout's rule matcher (one warp per rule, writes
// into shared SET / CLEAR), and ORs those into the global SET / CLEAR with
// atomics -- bands overlap in their last rows, whose writes merge there.
// After the last band the whole board combines (a bit changes where any
// match asks for it), the goal test and auto-reset run, and the next step's
// force plane is rebuilt from the player plane.
#include "launch.h"

namespace av {
namespace {

// Force plane word w for `action` from the player plane pl (plain words,
// nw of them): the player at p puts force at p + d (d = -W up, +1 right, +W
// down, -1 left), dropped where it would leave the board.
__device__ __forceinline__ uint32_t force_word(const DevConfig &cf, const uint32_t *pl, const uint32_t *masks,
                                               int nw, int w, int action)
{
    if (cf.ch_player < 0 || action < 1 || action > 4)
        return 0u;
    const int n = (action == 1 || action == 3) ? cf.W : 1;
    const int q = n >> 5, r = n & 31;
    uint32_t f = 0;
    if (action == 1 || action == 4) {  // toward lower p: bits [32w + n, 32w + n + 32)
        const uint32_t lo = w + q < nw ? pl[w + q] : 0u;
        const uint32_t hi = w + q + 1 < nw ? pl[w + q + 1] : 0u;
        f = __funnelshift_r(lo, hi, r);
    } else {  // toward higher p: bits [32w - n, 32w - n + 32)
        const int j = w - q;
        if (j >= 1)
            f = __funnelshift_l(pl[j - 1], pl[j], r);
        else if (j == 0)
            f = pl[0] << r;
    }
    if (action == 2)
        f &= ~masks[w];  // not from the last column onto the first
    else if (action == 4)
        f &= ~masks[nw + w];
    return f & masks[2 * nw + w];
}

template <typename CellT, int NA, bool SM>
__global__ void __launch_bounds__(kThreads)
    rollout_band_kernel(DevConfig cf, int band_rows, int band_nw, const uint32_t *__restrict__ arena,
                        const uint32_t *__restrict__ tab_off, const uint32_t *__restrict__ vm_g,
                        const uint32_t *__restrict__ masks_g, CellT *cur, const CellT *__restrict__ init,
                        int32_t *tsteps, int n_steps, uint64_t seed, const uint8_t *__restrict__ actions,
                        CellT *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
                        uint32_t *status, uint32_t *planes_g, uint32_t *set_g, uint32_t *clr_g, uint32_t *base_g)
{
    extern __shared__ __align__(16) unsigned char smem[];
    DevConfig bc = cf;  // the band as the rule matcher sees it
    bc.NW = band_nw;
    const Smem S = carve(smem, bc, 0);
    const int env = blockIdx.x, tid = threadIdx.x;
    const int H = cf.H, W = cf.W, HW = cf.HW, NW = cf.NW, NWP = cf.NWP, C = cf.C, NWB = band_nw;
    const int table = cf.rules_per_env ? env : 0;
    const uint32_t *tab_g = arena + tab_off[table];
    const uint32_t *tab = SM ? S.rules : tab_g;
    uint32_t *P = planes_g + (size_t)env * (C + 1) * NW;  // tiles 0..C-1, force C
    uint32_t *SETg = set_g + (size_t)env * C * NW;
    uint32_t *CLRg = clr_g + (size_t)env * C * NW;
    uint32_t *BASE = base_g + (size_t)env * C * NW;
    __shared__ int s_any;

    // ---- stage: shared planes zeroed once (entries past a band's words stay
    // zero), rule table, actions; the board and its initial map as planes
    for (int i = tid; i < (C + 1) * NWP; i += kThreads)
        S.planes[i] = make_uint2(0u, 0u);
    if (SM)
        stage_rules(tab_g, tab_off[table + 1] - tab_off[table], S.rules);
    if (tid < kWarps + 16)
        S.red[tid] = 0;
    fill_actions(actions, seed, env, 0, n_steps, S);
    const CellT *src = cur + (size_t)env * HW, *isrc = init + (size_t)env * HW;
    for (int w = tid; w < NW; w += kThreads) {
        uint32_t v[16], vi[16];
        for (int c = 0; c < C; ++c)
            v[c] = vi[c] = 0u;
        for (int b = 0; b < 32 && 32 * w + b < HW; ++b) {
            const uint32_t x = (uint32_t)src[32 * w + b], xi = (uint32_t)isrc[32 * w + b];
            for (int c = 0; c < C; ++c) {
                v[c] |= ((x >> c) & 1u) << b;
                vi[c] |= ((xi >> c) & 1u) << b;
            }
        }
        for (int c = 0; c < C; ++c) {
            P[c * NW + w] = v[c];
            BASE[c * NW + w] = vi[c];
            SETg[c * NW + w] = 0u;
            CLRg[c * NW + w] = 0u;
        }
    }
    __syncthreads();
    for (int w = tid; w < NW; w += kThreads)
        P[C * NW + w] = force_word(cf, P + (cf.ch_player >= 0 ? cf.ch_player : 0) * NW, masks_g, NW, w, S.acts[0]);
    if (tid == 0)
        S.flags[5] = S.acts[0];  // the action of the coming step (the ring slot may be refilled)
    int t = tsteps[env];
    int sum = 0;
    int goal_left = 1;  // of the board in hand, once a step has been evaluated on it
    __shared__ int s_chg;
    __syncthreads();

    // While the board stays as it is, the step with action a always has the
    // same outcome: an action whose step changed nothing is remembered (bit a
    // of S.flags[4], its reward in S.flags[8 + a]) and its later steps skip the
    // bands until the board changes or resets.
    const int n_bands = (H + band_rows - 1) / band_rows;
    const int warp = tid >> 5, lane = tid & 31;
    for (int s = 0; s < n_steps; ++s) {
        const bool refill = ((s + 1) & (kActChunk - 1)) == 0;
        if (refill)
            fill_actions(actions, seed, env, s + 1, n_steps, S);
        // A run of repeated steps, as in the block rollout: from this step on,
        // the steps whose actions are remembered and that end no episode with
        // an auto-reset take their remembered rewards, up to 32 at a time (lane
        // l of warp 0 takes step s + l), never up to the last step of the action
        // ring's chunk.  Warp 0 publishes the run's length and the next step's
        // action (S.flags[6], [7]) before a barrier that every thread reaches
        // after reading this step's action; the next force plane and S.flags[5]
        // are written after it, and a second barrier ends the run.
        if ((S.flags[4] >> S.flags[5]) & 1) {  // block-uniform
            if (refill)
                __syncthreads();  // the ring's next chunk
            if (warp == 0) {
                const int lim = min(min(32, n_steps - s), ((s + 1) | (kActChunk - 1)) - s);
                const int a_l = lane == 0 ? S.flags[5] : lane < lim ? (int)S.acts[(s + lane) & (kActChunk - 1)] : 0;
                const bool done_l = !goal_left || (cf.max_steps > 0 && t + lane + 1 >= cf.max_steps);
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
                sum += __reduce_add_sync(0xffffffffu, r_l);  // (thread 0's sum is the one kept)
                int a_next = __shfl_sync(0xffffffffu, a_l, e & 31);
                if (e == lim && s + e < n_steps)
                    a_next = S.acts[(s + e) & (kActChunk - 1)];
                if (lane == 0) {
                    S.flags[6] = e;
                    S.flags[7] = a_next;
                }
            }
            __syncthreads();
            const int e = S.flags[6];
            if (e > 0) {
                t += e;
                if (s + e < n_steps) {
                    const int a = S.flags[7];
                    for (int w = tid; w < NW; w += kThreads)
                        P[C * NW + w] =
                            force_word(cf, P + (cf.ch_player >= 0 ? cf.ch_player : 0) * NW, masks_g, NW, w, a);
                    if (tid == 0)
                        S.flags[5] = a;
                }
                if (obs_traj) {
                    for (int p = tid; p < HW; p += kThreads) {
                        uint32_t v = 0;
                        for (int c = 0; c < C; ++c)
                            v |= ((P[c * NW + (p >> 5)] >> (p & 31)) & 1u) << c;
                        for (int k = 0; k < e; ++k)
                            obs_traj[((size_t)(s + k) * cf.B + env) * HW + p] = (CellT)v;
                    }
                }
                __syncthreads();
                s += e - 1;
                continue;
            }
        }
        const int act = S.flags[5];
        const bool known = (S.flags[4] >> act) & 1;  // block-uniform (written before the last barrier)
        int rew = 0;
        for (int band = 0; known ? false : band < n_bands; ++band) {
            const int A0 = band * band_rows * W, A1 = min(H, (band + 1) * band_rows) * W;  // anchor cells
            const int w0 = A0 >> 5;
            for (int i = tid; i < (C + 1) * NWB; i += kThreads) {
                const int c = i / NWB, a = i - c * NWB;
                const uint32_t v = w0 + a < NW ? P[c * NW + w0 + a] : 0u;
                put_word(S.planes, NWP, c, a, v);
            }
            for (int i = tid; i < kShapes * NWB; i += kThreads) {
                const int shape = i / NWB, a = i - shape * NWB;
                const int g = w0 + a;
                uint32_t v = g < NW ? vm_g[(size_t)shape * NW + g] : 0u;
                const int lo = max(A0 - 32 * g, 0), hi = min(A1 - 32 * g, 32);  // band anchors in this word
                const uint32_t keep = lo >= hi ? 0u : ((hi == 32 ? 0xffffffffu : ((1u << hi) - 1u)) & ~((1u << lo) - 1u));
                S.vm[i] = v & keep;
            }
            for (int i = tid; i < C * NWB; i += kThreads) {
                S.setp[i] = 0u;
                S.clrp[i] = 0u;
            }
            __syncthreads();
            match_all<NA, SM>(bc, tab, S);
            __syncthreads();
            if (S.flags[0]) {
                for (int i = tid; i < C * NWB; i += kThreads) {
                    const int c = i / NWB, a = i - c * NWB;
                    if (w0 + a >= NW)
                        continue;
                    const uint32_t st = S.setp[i], cl = S.clrp[i];
                    if (st)
                        atomicOr(&SETg[c * NW + w0 + a], st);
                    if (cl)
                        atomicOr(&CLRg[c * NW + w0 + a], cl);
                }
            }
            if (tid < kWarps)
                rew += S.red[tid];  // thread w keeps warp w's band rewards
            __syncthreads();  // the shared band may be overwritten
            if (tid == 0)
                S.flags[0] = 0;
        }
        // ---- the whole board: combine, goal test, reset, next force plane
        if (!known) {
            if (tid == 0) {
                s_any = 0;
                s_chg = 0;
            }
            __syncthreads();
            int goal = 0, chg = 0;
            for (int i = tid; i < C * NW; i += kThreads) {
                uint32_t d = P[i];
                const uint32_t st = SETg[i], cl = CLRg[i];
                if (st | cl) {
                    const uint32_t nd = (d & ~cl) | (~d & st);
                    chg |= nd != d;
                    d = nd;
                    P[i] = d;
                    SETg[i] = 0u;
                    CLRg[i] = 0u;
                }
                if (cf.ch_goal >= 0 && i / NW == cf.ch_goal && d)
                    goal = 1;
            }
            if (goal)
                s_any = 1;
            if (chg)
                s_chg = 1;
            rew = __reduce_add_sync(0xffffffffu, rew);  // warp 0 holds every warp's share
            if (tid == 0)
                S.flags[3] = rew;
            __syncthreads();
            goal_left = cf.ch_goal < 0 || s_any;
            if (tid == 0) {  // remember the step if it left the board as it was
                if (s_chg) {
                    S.flags[4] = 0;
                } else {
                    S.flags[4] |= 1 << act;
                    S.flags[8 + act] = rew;
                }
            }
        }
        t += 1;
        const int done = !goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
        if (done && cf.auto_reset) {
            for (int i = tid; i < C * NW; i += kThreads)
                P[i] = BASE[i];
            t = 0;
            if (tid == 0)
                S.flags[4] = 0;  // the board may have changed
        }
        const int step_rew = known ? S.flags[8 + act] : S.flags[3];
        sum += step_rew;
        if (tid == 0) {
            if (rew_traj)
                rew_traj[(size_t)s * cf.B + env] = step_rew;
            if (done_traj)
                done_traj[(size_t)s * cf.B + env] = (uint8_t)done;
        }
        __syncthreads();  // the board after any reset
        if (s + 1 < n_steps) {
            const int a = S.acts[(s + 1) & (kActChunk - 1)];
            for (int w = tid; w < NW; w += kThreads)
                P[C * NW + w] = force_word(cf, P + (cf.ch_player >= 0 ? cf.ch_player : 0) * NW, masks_g, NW, w, a);
            if (tid == 0)
                S.flags[5] = a;
        }
        if (obs_traj) {
            CellT *o = obs_traj + ((size_t)s * cf.B + env) * HW;
            for (int p = tid; p < HW; p += kThreads) {
                uint32_t v = 0;
                for (int c = 0; c < C; ++c)
                    v |= ((P[c * NW + (p >> 5)] >> (p & 31)) & 1u) << c;
                o[p] = (CellT)v;
            }
        }
        __syncthreads();
    }
    CellT *dst = cur + (size_t)env * HW;
    for (int p = tid; p < HW; p += kThreads) {
        uint32_t v = 0;
        for (int c = 0; c < C; ++c)
            v |= ((P[c * NW + (p >> 5)] >> (p & 31)) & 1u) << c;
        dst[p] = (CellT)v;
    }
    if (tid == 0) {
        tsteps[env] = t;
        if (rew_sum)
            rew_sum[env] = sum;
        if (S.flags[1])
            atomicOr(status + 1, kWarnAction);
    }
}

#define AV_FOR_NA(MACRO, CELL) MACRO(CELL, 1) MACRO(CELL, 2) MACRO(CELL, 4) MACRO(CELL, 8) MACRO(CELL, 16)

template <typename CellT, int NA>
void band_t(const DevConfig &cf, int band_rows, int band_nw, const uint32_t *arena, const uint32_t *tab_off,
            const uint32_t *vm, const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps,
            uint64_t seed, const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj,
            int32_t *rew_sum, uint32_t *status, uint32_t *planes, uint32_t *set, uint32_t *clr, uint32_t *base,
            cudaStream_t st)
{
    DevConfig bc = cf;
    bc.NW = band_nw;
    const size_t sm = step_smem(bc, 0).total;
    if (cf.rule_words > 0)
        rollout_band_kernel<CellT, NA, true><<<cf.B, kThreads, sm, st>>>(
            cf, band_rows, band_nw, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed,
            actions, (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status, planes, set, clr, base);
    else
        rollout_band_kernel<CellT, NA, false><<<cf.B, kThreads, sm, st>>>(
            cf, band_rows, band_nw, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed,
            actions, (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status, planes, set, clr, base);
}

}  // namespace

cudaError_t configure_band()
{
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    };
#define AV_SET(CELL, NA)                                     \
    set((const void *)rollout_band_kernel<CELL, NA, true>);  \
    set((const void *)rollout_band_kernel<CELL, NA, false>);
    AV_FOR_NA(AV_SET, uint8_t)
    AV_FOR_NA(AV_SET, uint16_t)
#undef AV_SET
    return e;
}

void band_geometry(int H, int W, int *band_rows, int *band_nw, int *na, int *nwp)
{
    // the most rows whose anchors and the four rows below them fit 128 words
    // (with a word of slack on each side), so that the block matcher's lanes
    // (8 x NA words, NA <= 16) cover the band
    int rows = H;
    auto words = [&](int r) { return (31 + r * W + 4 * W + 4 + 31) / 32 + 1; };
    while (rows > 1 && words(rows) > 128)
        --rows;
    *band_rows = rows;
    *band_nw = words(rows);
    int a = 1;
    while (8 * a < *band_nw)
        a *= 2;
    *na = a;
    *nwp = 8 * a + (4 * W + 4) / 32 + 2;  // a lane's words plus the farthest term offset
}

void launch_rollout_band(const DevConfig &cf, int band_rows, int band_nw, const uint32_t *arena,
                         const uint32_t *tab_off, const uint32_t *vm, const uint32_t *masks, void *cur,
                         const void *init, int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions,
                         void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                         uint32_t *planes, uint32_t *set, uint32_t *clr, uint32_t *base, cudaStream_t st)
{
#define AV_CASE(CELL, NA)                                                                                         \
    case NA:                                                                                                     \
        band_t<CELL, NA>(cf, band_rows, band_nw, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, \
                         obs_traj, rew_traj, done_traj, rew_sum, status, planes, set, clr, base, st);              \
        break;
    if (cf.cell_bytes == 1) {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint8_t) }
    } else {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint16_t) }
    }
#undef AV_CASE
}

}  // namespace av
