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

// Outputs of the kept matches into SET / CLEAR; returns this lane's reward.
template <int NA, bool SM>
__device__ __forceinline__ int write_matches(const DevConfig &cf, const uint32_t *tab, int r, const Smem &S,
                                             const uint32_t (&m)[NA])
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
            scatter_bits(S.setp, ov.z, cf.NW, w0, lo, hi);
            scatter_bits(S.clrp, ov.w, cf.NW, w0, lo, hi);
        }
    }
    S.flags[0] = 1;
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
            rew += write_matches<NA, SM>(cf, tab, r, S, m);
        }
        rew = __reduce_add_sync(0xffffffffu, rew);
        if (lane == 0)
            S.red[warp] = rew;
        __syncthreads();
        if (warp == 0) {
            // combine: a bit changes where any kept match asks for it
            if (S.flags[0]) {
                for (int c = 0; c < C; ++c)
                    for (int w = lane; w < NW; w += 32) {
                        const int i = c * NW + w;
                        const uint32_t d = S.planes[c * NWP + w].x, st = S.setp[i], cl = S.clrp[i];
                        S.setp[i] = 0u;
                        S.clrp[i] = 0u;
                        put_word(S.planes, NWP, c, w, (d & ~cl) | (~d & st));
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
                for (int c = 0; c < C; ++c)
                    for (int w = lane; w < NW; w += 32)
                        put_word(S.planes, NWP, c, w, S.basep[c * NW + w]);
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
    return e;
}

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
    if (cf.cell_bytes == 1) {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint8_t) }
    } else {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint16_t) }
    }
#undef AV_CASE
}

}  // namespace av
