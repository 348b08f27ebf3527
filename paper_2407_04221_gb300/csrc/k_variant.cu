// k_variant.cu -- rollouts under the variant rule semantics sketched at the end
// of Sec. 2.1 ("Possible extensions"): a rule applied only once or a fixed
// number of times per step, the tiles to rewrite chosen by the maximum over an
// ordered or random index channel; rules inhibiting others by masking.
//
// A match is (rule r, rotation g, anchor cell p); its key is (p << 2) | g, or
// with random indices ((draw(key_seed, 13, env, t, p) >> 48) << 14) | (p << 2)
// | g, t the env's step counter before the step.  limit[r] = k > 0 keeps the
// k matches of rule r with the largest keys; a rule with any raw match this
// step suppresses the rules of its inhibit mask (decided on raw matches, so
// rule order does not matter).
//
// One CTA of kThreads per environment, boards staged as bit-planes as in the
// block rollout kernel.  Each step runs two passes over the rules, one warp
// per rule: pass 1 finds which rules have a raw match; after a barrier every
// warp derives the suppressed set; pass 2 re-evaluates the rules that matched
// and are not suppressed, keeps the largest keys by warp max-reductions when
// the rule is limited, and writes the kept matches' outputs.  The combine,
// goal test and auto-reset are those of the standard step.
#include "launch.h"

namespace av {
namespace {

// Anchors of rule r in this lane's rotation (lane >> 3) and words
// (lane & 7) + 8u where every term holds.  Returns whether any lane has one
// (warp-uniform); stops early once none is left.
template <int NA, bool SM>
__device__ __forceinline__ bool rule_matches(const DevConfig &cf, const uint32_t *tab, int r, const Smem &S,
                                             uint32_t (&m)[NA])
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    const uint4 h0 = ld4<SM>(tab + 4 + 8 * r);  // n_present, n_absent, n_out, reward
    const uint4 h1 = ld4<SM>(tab + 8 + 8 * r);  // first term, first output, shapes
    const uint32_t *vmr = S.vm + ((h1.z >> (8 * g)) & 0xffu) * cf.NW;
#pragma unroll
    for (int u = 0; u < NA; ++u) {
        const int a = q + 8 * u;
        m[u] = a < cf.NW ? vmr[a] : 0u;
    }
    const uint2 *tp = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R)) + (size_t)h1.x * 4 + g;
    const unsigned char *pb = reinterpret_cast<const unsigned char *>(S.planes) + q * 8;
    const uint32_t nt = h0.x + h0.y;
    for (uint32_t t = 0; t < nt; ++t) {
        const uint2 d = ld2<SM>(tp + 4 * t);
        const uint32_t neg = (uint32_t)((int32_t)d.y >> 31);  // absent term: complement
        uint32_t any = 0;
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            const uint2 w = *reinterpret_cast<const uint2 *>(pb + d.x + 64 * u);
            m[u] &= __funnelshift_r(w.x, w.y, d.y) ^ neg;
            any |= m[u];
        }
        if ((t & 1u) && !__any_sync(0xffffffffu, any != 0u))
            return false;
    }
    uint32_t any = 0;
#pragma unroll
    for (int u = 0; u < NA; ++u)
        any |= m[u];
    return __any_sync(0xffffffffu, any != 0u);
}

// Key of the match at anchor cell p in rotation g (see the file comment);
// keys are below 2^30 and distinct within a rule.
__device__ __forceinline__ uint32_t match_key(const VariantParams &vp, int env, int t, uint32_t p, uint32_t g)
{
    uint32_t key = (p << 2) | g;
    if (vp.random_keys)
        key |= (uint32_t)(draw(vp.key_seed, 13, (uint64_t)env, (uint64_t)(uint32_t)t, p) >> 48) << 14;
    return key;
}

// Keep only the k matches of m with the largest keys (one warp).
template <int NA>
__device__ __forceinline__ void keep_largest(uint32_t (&m)[NA], int k, const VariantParams &vp, int env, int t)
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    uint32_t kept[NA];
#pragma unroll
    for (int u = 0; u < NA; ++u)
        kept[u] = 0u;
    for (int i = 0; i < k; ++i) {
        uint32_t best = 0;  // this lane's largest key + 1 (0: no candidate left)
        int bu = 0, bb = 0;
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            const uint32_t base = (uint32_t)(q + 8 * u) * 32u;
            if (!vp.random_keys) {
                if (m[u]) {  // the highest anchor of the highest word wins
                    const int b = 31 - __clz(m[u]);
                    best = ((base + (uint32_t)b) << 2 | (uint32_t)g) + 1u;
                    bu = u;
                    bb = b;
                }
            } else {
                for (uint32_t x = m[u]; x; x &= x - 1u) {
                    const int b = __ffs(x) - 1;
                    const uint32_t key = match_key(vp, env, t, base + (uint32_t)b, (uint32_t)g) + 1u;
                    if (key > best) {
                        best = key;
                        bu = u;
                        bb = b;
                    }
                }
            }
        }
        const uint32_t top = __reduce_max_sync(0xffffffffu, best);
        if (top == 0u)
            break;
        if (best == top) {  // keys are distinct: exactly one lane
#pragma unroll
            for (int u = 0; u < NA; ++u)
                if (u == bu) {
                    kept[u] |= 1u << bb;
                    m[u] &= ~(1u << bb);
                }
        }
    }
#pragma unroll
    for (int u = 0; u < NA; ++u)
        m[u] = kept[u];
}

// Outputs of the kept matches into SET / CLEAR (setp / clrp, NW words per
// channel); returns this lane's reward.
template <int NA, bool SM>
__device__ __forceinline__ int write_matches(const DevConfig &cf, const uint32_t *tab, int r, uint32_t *setp,
                                             uint32_t *clrp, const uint32_t (&m)[NA])
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    uint32_t cnt = 0;
#pragma unroll
    for (int u = 0; u < NA; ++u)
        cnt += __popc(m[u]);
    if (cnt == 0)
        return 0;
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
    return (int)h0.w * (int)cnt;
}

template <typename CellT, int NA, bool SM>
__global__ void __launch_bounds__(kThreads)
    rollout_variant_kernel(DevConfig cf, const __grid_constant__ VariantParams vp,
                           const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
                           const uint32_t *__restrict__ vm_g, const uint32_t *__restrict__ masks_g, CellT *cur,
                           const CellT *__restrict__ init, int32_t *tsteps, int n_steps, uint64_t seed,
                           const uint8_t *__restrict__ actions, CellT *obs_traj, int32_t *rew_traj,
                           uint8_t *done_traj, int32_t *rew_sum, uint32_t *status)
{
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ uint32_t s_raw[2];  // rules with a raw match this step
    __shared__ int s_t;            // the env's step counter
    const Smem S = carve(smem, cf, 0);
    const int env = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int HW = cf.HW, NW = cf.NW, NWP = cf.NWP, C = cf.C;
    const int table = cf.rules_per_env ? env : 0;
    const uint32_t *tab_g = arena + tab_off[table];
    const uint32_t *tab = SM ? S.rules : tab_g;

    stage_common(cf, S, vm_g, masks_g);
    if (SM)
        stage_rules(tab_g, tab_off[table + 1] - tab_off[table], S.rules);
    if (tid == 0) {
        s_raw[0] = s_raw[1] = 0u;
        s_t = tsteps[env];
    }
    __syncthreads();
    cells_to_planes<CellT>(cf, cur + (size_t)env * HW, S.planes, nullptr);
    cells_to_planes<CellT>(cf, init + (size_t)env * HW, nullptr, S.basep);
    fill_actions(actions, seed, env, 0, n_steps, S);
    __syncthreads();
    if (warp == 0)
        write_force(cf, S, S.acts[0]);
    __syncthreads();

    int sum = 0;
    for (int s = 0; s < n_steps; ++s) {
        if (((s + 1) & (kActChunk - 1)) == 0)
            fill_actions(actions, seed, env, s + 1, n_steps, S);
        const int t = s_t;
        // pass 1: which rules have a raw match
        for (int r = warp; r < cf.R; r += kWarps) {
            uint32_t m[NA];
            if (rule_matches<NA, SM>(cf, tab, r, S, m) && lane == 0)
                atomicOr(&s_raw[r >> 5], 1u << (r & 31));
        }
        __syncthreads();
        const uint64_t raw = (uint64_t)s_raw[0] | ((uint64_t)s_raw[1] << 32);
        uint64_t sup = 0;
        for (uint64_t x = raw; x; x &= x - 1u)
            sup |= vp.inhibit[__ffsll((long long)x) - 1];
        // pass 2: the rules that apply, their kept matches written
        int rew = 0;
        for (int r = warp; r < cf.R; r += kWarps) {
            if (!((raw >> r) & 1u) || ((sup >> r) & 1u))
                continue;
            uint32_t m[NA];
            rule_matches<NA, SM>(cf, tab, r, S, m);
            if (vp.limit[r] > 0)
                keep_largest<NA>(m, vp.limit[r], vp, env, t);
            uint32_t kept = 0;
#pragma unroll
            for (int u = 0; u < NA; ++u)
                kept |= m[u];
            if (kept)
                S.flags[0] = 1;  // this lane writes
            rew += write_matches<NA, SM>(cf, tab, r, S.setp, S.clrp, m);
        }
        rew = __reduce_add_sync(0xffffffffu, rew);
        if (lane == 0)
            S.red[warp] = rew;
        __syncthreads();
        if (warp == 0) {
            // combine: a bit changes where any kept match asks for it
            if (S.flags[0]) {
                // one index over every channel's words; (c, w) stepped without a division
                for (int i = lane, c = lane / NW, w = lane - (lane / NW) * NW; i < C * NW; i += 32) {
                    const uint32_t d = S.planes[c * NWP + w].x, st = S.setp[i], cl = S.clrp[i];
                    S.setp[i] = 0u;
                    S.clrp[i] = 0u;
                    put_word(S.planes, NWP, c, w, (d & ~cl) | (~d & st));
                    for (w += 32; w >= NW; w -= NW)
                        ++c;
                }
                __syncwarp();
                if (lane == 0)
                    S.flags[0] = 0;
            }
            int goal = cf.ch_goal < 0;
            if (cf.ch_goal >= 0)
                for (int w = lane; w < NW; w += 32)
                    goal |= S.planes[cf.ch_goal * NWP + w].x != 0u;
            goal = __any_sync(0xffffffffu, goal);
            int tn = t + 1;
            const int done = !goal || (cf.max_steps > 0 && tn >= cf.max_steps);
            if (done && cf.auto_reset) {
                for (int i = lane, c = lane / NW, w = lane - (lane / NW) * NW; i < C * NW; i += 32) {
                    put_word(S.planes, NWP, c, w, S.basep[i]);
                    for (w += 32; w >= NW; w -= NW)
                        ++c;
                }
                tn = 0;
            }
            int total = lane < kWarps ? S.red[lane] : 0;
            total = __reduce_add_sync(0xffffffffu, total);
            sum += total;
            if (lane == 0) {
                if (rew_traj)
                    rew_traj[(size_t)s * cf.B + env] = total;
                if (done_traj)
                    done_traj[(size_t)s * cf.B + env] = (uint8_t)done;
                s_t = tn;
                s_raw[0] = s_raw[1] = 0u;
            }
            __syncwarp();
            if (s + 1 < n_steps)
                write_force(cf, S, S.acts[(s + 1) & (kActChunk - 1)]);
        }
        __syncthreads();
        if (obs_traj)
            store_cells<CellT>(cf, S.planes, obs_traj + ((size_t)s * cf.B + env) * HW, tid, kThreads);
    }
    store_cells<CellT>(cf, S.planes, cur + (size_t)env * HW, tid, kThreads);
    if (tid == 0) {
        tsteps[env] = s_t;
        if (rew_sum)
            rew_sum[env] = sum;
        if (S.flags[1])
            atomicOr(status + 1, kWarnAction);
    }
}

// The remaining terms of a rule after its register-resident ones (padded
// batches, as the one-warp rollout evaluates them), ANDed into m; no write.
template <int NA, bool SM>
__device__ __forceinline__ void rest_terms(const DevConfig &cf, const uint32_t *tab, uint32_t pbase, uint32_t rest,
                                           uint32_t (&m)[NA])
{
    const uint2 *tp = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R)) + (rest >> 8);
    const uint32_t nb = rest & 0xffu;
    for (uint32_t b = 0; b < nb; ++b, tp += 4 * kRestBatch) {
        uint2 d[kRestBatch];
#pragma unroll
        for (int j = 0; j < kRestBatch; ++j)
            d[j] = ld2<SM>(tp + 4 * j);
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            uint32_t x = 0xffffffffu;
#pragma unroll
            for (int j = 0; j < kRestBatch; ++j) {
                const uint2 w = lds2(pbase + d[j].x + 64 * u);
                x &= __funnelshift_r(w.x, w.y, d[j].y) ^ (uint32_t)((int32_t)d[j].y >> 31);
            }
            m[u] &= x;
        }
    }
}

// One warp per environment (boards of at most 512 cells, at most 16 rules),
// on the one-warp rollout's layout and loop: each lane keeps every rule's
// first four present terms in registers, and a step in which no rule
// survives them has no raw match, so it is the standard quiet step; nor has a
// rule whose tile terms pass nowhere on the board (tested once per board).  A
// step with survivors finishes their remaining terms into the registers (no
// writes yet: the raw matches), derives the suppressed set, keeps each
// limited rule's largest keys, writes, and updates the board; no barrier.
template <typename CellT, int NA, int RPW, bool SM>
__global__ void __launch_bounds__(128)
    rollout_variant_warp_kernel(DevConfig cf, const __grid_constant__ VariantParams vp,
                                const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
                                const uint32_t *__restrict__ vm_g, const uint32_t *__restrict__ masks_g,
                                CellT *cur, const CellT *__restrict__ init, int32_t *tsteps, int n_steps,
                                uint64_t seed, const uint8_t *__restrict__ actions, CellT *obs_traj,
                                int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status)
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
    const uint32_t ones = (uint32_t)(C + 6) * (uint32_t)NWP * 8;  // the all-ones plane
    uint2 *const slot = S.planes + C * NWP;
    const uint2 *const fplanes = S.planes + (C + 1) * NWP;

    // ---- stage (this warp's environment only), as the one-warp rollout does
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
    for (int k = lane; k < kActChunk; k += 32)
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

    // ---- per-lane register data of every rule (its first four present terms)
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
                    if ((uint32_t)j < h0.x) {
                        const uint2 d = ld2<SM>(terms + (size_t)(h1.x + j) * 4 + g);
                        f.a[j] = pbase + d.x;
                        f.s[j] = d.y;
                    }
                const uint32_t t0 = min(h0.x, (uint32_t)kRegTerms);
                const uint32_t nb = (h0.x + h0.y - t0 + kRestBatch - 1) / kRestBatch;
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
    __syncwarp();
    const bool any_traj = rew_traj != nullptr || done_traj != nullptr || obs_traj != nullptr;

    int sum = 0;
    // Rules tested on the current board and those that cannot match on it
    // (env_dead_rules; warp-uniform, cleared when the board changes), and per
    // rule a mask that is zero for such a rule, applied to the step's first vote
    // (kernels with more than eight rules per lane skip that vote: their
    // registers are full already).
    constexpr bool kQuietVote = RPW <= 8;
    uint32_t known = 0, dead = 0;
    uint32_t alive[kQuietVote ? RPW : 1];
#pragma unroll
    for (int k = 0; k < (kQuietVote ? RPW : 1); ++k)
        alive[k] = 0xffffffffu;
    for (int s = 0; s < n_steps; ++s) {
        if (s > 0 && (s & (kActChunk / 2 - 1)) == 0)
            env_refill(actions, seed, env, s, n_steps, S.acts, S.ctl + 3);
        const int a_next = S.acts[(s + 1) & (kActChunk - 1)];
        uint32_t m[RPW][NA];
        uint32_t anyall = 0;
#pragma unroll
        for (int k = 0; k < RPW; ++k)
#pragma unroll
            for (int u = 0; u < NA; ++u) {
                m[k][u] = env_reg_terms(fr[k], u);
                anyall |= m[k][u] & alive[kQuietVote ? k : 0];
            }
        uint32_t live = 0;
        if (!kQuietVote || __any_sync(0xffffffffu, anyall != 0u)) {  // else a quiet step
            uint32_t bits = 0;
#pragma unroll
            for (int k = 0; k < RPW; ++k) {
                uint32_t a = 0;
#pragma unroll
                for (int u = 0; u < NA; ++u)
                    a |= m[k][u];
                bits |= (a != 0u ? 1u : 0u) << k;
            }
            live = __reduce_or_sync(0xffffffffu, bits);  // rules past their register terms
            if (live & ~known) {  // rules live for the first time on this board
                dead |= env_dead_rules<NA, SM>(cf, tab, S.vm, pbase, live & ~known);
                known |= live;
#pragma unroll
                for (int k = 0; k < (kQuietVote ? RPW : 1); ++k)
                    alive[k] = ((dead >> k) & 1u) ? 0u : 0xffffffffu;
            }
            live &= ~dead;  // no raw match possible: neither written nor inhibiting
        }
        int rew = 0, changed = 0;
        if (live) {
            // raw matches: the rest of every live rule, into m (no writes)
            uint32_t raw = 0;
#pragma unroll
            for (int k = 0; k < RPW; ++k)
                if ((live >> k) & 1u) {
                    rest_terms<NA, SM>(cf, tab, pbase, fr[k].rest, m[k]);
                    uint32_t a = 0;
#pragma unroll
                    for (int u = 0; u < NA; ++u)
                        a |= m[k][u];
                    if (__any_sync(0xffffffffu, a != 0u))
                        raw |= 1u << k;
                }
            uint64_t sup = 0;
            for (uint32_t x = raw; x; x &= x - 1u)
                sup |= vp.inhibit[__ffs(x) - 1];
            uint32_t wrote = 0;
#pragma unroll
            for (int k = 0; k < RPW; ++k) {
                if (!((raw >> k) & 1u) || ((sup >> k) & 1u))
                    continue;
                if (vp.limit[k] > 0)
                    keep_largest<NA>(m[k], vp.limit[k], vp, env, t);
#pragma unroll
                for (int u = 0; u < NA; ++u)
                    wrote |= m[k][u];
                rew += write_matches<NA, SM>(cf, tab, k, S.setp, S.clrp, m[k]);
            }
            rew = __reduce_add_sync(0xffffffffu, rew);
            changed = __any_sync(0xffffffffu, wrote != 0u);
        }
        t += 1;
        int done = !goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
        if (changed || (done && cf.auto_reset)) {
            const int3 r = env_board_update(cf, S.planes, S.setp, S.clrp, S.basep, S.masks, t);
            t = r.x;
            goal_left = r.y;
            done = r.z;
            known = 0;  // a new board
            dead = 0;
#pragma unroll
            for (int k = 0; k < (kQuietVote ? RPW : 1); ++k)
                alive[k] = 0xffffffffu;
        }
        sum += rew;
        // every read of this step's force is behind the step's last vote
        if (lane < NW)
            slot[lane] = fplanes[a_next * NWP + lane];
        __syncwarp();
        if (any_traj)
            env_step_outputs<CellT>(cf, S.planes, env, s, rew, done, obs_traj, rew_traj, done_traj);
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

#define AV_FOR_NA(MACRO, CELL) MACRO(CELL, 1) MACRO(CELL, 2) MACRO(CELL, 4) MACRO(CELL, 8) MACRO(CELL, 16)

template <typename CellT, int NA>
void variant_t(const DevConfig &cf, const VariantParams &vp, const uint32_t *arena, const uint32_t *tab_off,
               const uint32_t *vm, const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps,
               uint64_t seed, const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj,
               int32_t *rew_sum, uint32_t *status, cudaStream_t st)
{
    const size_t sm = step_smem(cf, 0).total;
    if (cf.rule_words > 0)
        rollout_variant_kernel<CellT, NA, true><<<cf.B, kThreads, sm, st>>>(
            cf, vp, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
            (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
    else
        rollout_variant_kernel<CellT, NA, false><<<cf.B, kThreads, sm, st>>>(
            cf, vp, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
            (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
}

template <typename CellT, int NA, int RPW>
void variant_warp_t(const DevConfig &cf, const VariantParams &vp, const uint32_t *arena, const uint32_t *tab_off,
                    const uint32_t *vm, const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps,
                    uint64_t seed, const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj,
                    int32_t *rew_sum, uint32_t *status, cudaStream_t st)
{
    const int epb = env_warps_per_cta(cf);
    const size_t sm = (size_t)epb * fast_layout(cf).total;
    const int grid = (cf.B + epb - 1) / epb;
    if (cf.rule_words > 0)
        rollout_variant_warp_kernel<CellT, NA, RPW, true><<<grid, 32 * epb, sm, st>>>(
            cf, vp, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
            (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
    else
        rollout_variant_warp_kernel<CellT, NA, RPW, false><<<grid, 32 * epb, sm, st>>>(
            cf, vp, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
            (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
}

template <typename CellT, int NA>
void variant_warp_na(const DevConfig &cf, const VariantParams &vp, const uint32_t *arena, const uint32_t *tab_off,
                     const uint32_t *vm, const uint32_t *masks, void *cur, const void *init, int32_t *t,
                     int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj, int32_t *rew_traj,
                     uint8_t *done_traj, int32_t *rew_sum, uint32_t *status, cudaStream_t st)
{
#define AV_VW(RPW)                                                                                             \
    variant_warp_t<CellT, NA, RPW>(cf, vp, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj, \
                                   rew_traj, done_traj, rew_sum, status, st)
    if (cf.R <= 4) AV_VW(4);
    else if (cf.R <= 8) AV_VW(8);
    else AV_VW(16);
#undef AV_VW
}

}  // namespace

cudaError_t configure_variant()
{
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    };
#define AV_SET(CELL, NA)                                        \
    set((const void *)rollout_variant_kernel<CELL, NA, true>);  \
    set((const void *)rollout_variant_kernel<CELL, NA, false>);
    AV_FOR_NA(AV_SET, uint8_t)
    AV_FOR_NA(AV_SET, uint16_t)
#undef AV_SET
#define AV_SETW(CELL, NA, RPW)                                            \
    set((const void *)rollout_variant_warp_kernel<CELL, NA, RPW, true>);  \
    set((const void *)rollout_variant_warp_kernel<CELL, NA, RPW, false>);
#define AV_SETW_ALL(CELL, NA) AV_SETW(CELL, NA, 4) AV_SETW(CELL, NA, 8) AV_SETW(CELL, NA, 16)
    AV_SETW_ALL(uint8_t, 1)
    AV_SETW_ALL(uint8_t, 2)
    AV_SETW_ALL(uint16_t, 1)
    AV_SETW_ALL(uint16_t, 2)
#undef AV_SETW_ALL
#undef AV_SETW
    return e;
}

// One warp per environment for small boards with few rules whose rule set is
// not flagged busy (use_variant_warp), else one CTA per environment.
void launch_rollout_variant(const DevConfig &cf, const VariantParams &vp, const uint32_t *arena,
                            const uint32_t *tab_off, const uint32_t *vm, const uint32_t *masks, void *cur,
                            const void *init, int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions,
                            void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
                            uint32_t *status, cudaStream_t st)
{
#define AV_CASE(CELL, NA)                                                                                    \
    case NA:                                                                                                \
        variant_t<CELL, NA>(cf, vp, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj, \
                            rew_traj, done_traj, rew_sum, status, st);                                      \
        break;
    if (use_variant_warp(cf)) {
        if (cf.cell_bytes == 1 && cf.NA == 1)
            variant_warp_na<uint8_t, 1>(cf, vp, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                        obs_traj, rew_traj, done_traj, rew_sum, status, st);
        else if (cf.cell_bytes == 1)
            variant_warp_na<uint8_t, 2>(cf, vp, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                        obs_traj, rew_traj, done_traj, rew_sum, status, st);
        else if (cf.NA == 1)
            variant_warp_na<uint16_t, 1>(cf, vp, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                         obs_traj, rew_traj, done_traj, rew_sum, status, st);
        else
            variant_warp_na<uint16_t, 2>(cf, vp, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                         obs_traj, rew_traj, done_traj, rew_sum, status, st);
        return;
    }
    if (cf.cell_bytes == 1) {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint8_t) }
    } else {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint16_t) }
    }
#undef AV_CASE
}

}  // namespace av
