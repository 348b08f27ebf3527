// k_step.cu -- one step of every environment given its action (av_step), one
// warp per environment: the launch shape of single-step use, where no outcome
// can be repeated and a CTA's setup is most of the work.
//
// Each warp holds its environment's board as doubled bit-planes (tile
// channels 0..C-1, the force plane C, a zero plane C + 1 that the table's
// padding terms read as absent) and its own SET / CLEAR planes; the rule table
// is read where it lies (L1 / L2), not copied: a single step reads each term it
// tests once.  The warp tests every rule in its four rotations exactly as the
// other kernels do (Sec. 2.1, Eq. 2: lane = rotation x anchor word, four terms
// per vote, a rule left as soon as no anchor is live), ORs the outputs of live
// matches into SET / CLEAR (the transposed-convolution write, Eq. 3), pays
// reward x matches, combines next = (D & ~CLEAR) | (~D & SET), tests the goal,
// resets on done when asked to and writes the board, its observation, the
// reward, done flag and step counter.  Eight environments share a CTA and its
// copy of the valid-anchor and column masks; after staging those no warp waits
// for another.
#include "launch.h"

namespace av {
namespace {

constexpr int kStepWarps = 8;  // environments per CTA

struct StepWarpLayout {
    size_t vm, masks, warps;                   // CTA region
    size_t planes, setp, clrp, hdr, lead, per_warp;  // within a warp's region
    size_t total;
};

inline __host__ __device__ size_t align16s(size_t x) { return (x + 15) & ~(size_t)15; }

__host__ __device__ inline StepWarpLayout step_warp_layout(const DevConfig &cf)
{
    StepWarpLayout L;
    L.vm = 0;
    L.masks = align16s((size_t)kShapes * cf.NW * 4);
    L.warps = align16s(L.masks + (size_t)3 * cf.NW * 4);
    L.planes = 0;
    L.setp = align16s((size_t)(cf.C + 2) * cf.NWP * 8);
    L.clrp = align16s(L.setp + (size_t)cf.C * cf.NW * 4);
    L.hdr = align16s(L.clrp + (size_t)cf.C * cf.NW * 4);
    L.lead = align16s(L.hdr + (size_t)cf.R * 32);
    L.per_warp = align16s(L.lead + (size_t)cf.R * 4 * 4 * 8);
    L.total = L.warps + (size_t)kStepWarps * L.per_warp;
    return L;
}

// The outputs of one rule (n_out entries at `op`, this lane's rotation) at the
// live anchors m, ORed into this warp's SET / CLEAR planes.  Output entry at
// window offset s = 32 d + sh moves the anchors of word j to word j + d
// (shifted left by sh) and j + d + 1: the owner of word W takes
// (M[W - d] << sh) | (M[W - d - 1] >> (32 - sh)), fetching its rotation's match
// words by shuffles (word j of a rotation is lane (j & 7) of its quarter,
// anchor slot j >> 3); two xor-shuffles OR the four rotations, and the lanes of
// quarter 0 write each word (one lane per word; the planes are this warp's).
template <int NA>
__device__ __forceinline__ void step_write(const DevConfig &cf, const uint4 *op, uint32_t n_out,
                                           const uint32_t (&m)[NA], uint32_t *wset, uint32_t *wclr)
{
    const int lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    uint4 next = n_out ? __ldg(op) : make_uint4(0u, 0u, 0u, 0u);
    for (uint32_t o = 0; o < n_out; ++o) {
        const uint4 ov = next;
        if (o + 1 < n_out)  // the next entry's load overlaps this one's work
            next = __ldg(op + 4 * (o + 1));
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

// The board's cells from the doubled planes into dst and, when set, dst2
// (one warp; each cell word built once).
template <typename CellT>
__device__ __forceinline__ void step_store_cells(const DevConfig &cf, const uint2 *dbl, CellT *dst, CellT *dst2)
{
    constexpr int kPer = 4 / (int)sizeof(CellT);
    const int lane = threadIdx.x & 31, HW = cf.HW, NWP = cf.NWP;
    const int n_words = (HW + kPer - 1) / kPer;
    const bool aligned = (HW % kPer) == 0 && (reinterpret_cast<uintptr_t>(dst) & 3u) == 0 &&
                         (!dst2 || (reinterpret_cast<uintptr_t>(dst2) & 3u) == 0);
    for (int g = lane; g < n_words; g += 32) {
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
            if (dst2)
                reinterpret_cast<uint32_t *>(dst2)[g] = v;
        } else {
            for (int k = 0; k < kPer && p0 + k < HW; ++k) {
                dst[p0 + k] = (CellT)(v >> (8 * (int)sizeof(CellT) * k));
                if (dst2)
                    dst2[p0 + k] = (CellT)(v >> (8 * (int)sizeof(CellT) * k));
            }
        }
    }
}

// A board's cells (global) into the warp's doubled tile planes: per 32 cells
// one ballot per channel, lane c keeping channel c's word, then every channel
// written in one store (C <= 32).
template <typename CellT>
__device__ __forceinline__ void step_load_planes(const DevConfig &cf, const CellT *__restrict__ src, uint2 *dbl)
{
    const int lane = threadIdx.x & 31;
    for (int base = 0; base < cf.HW; base += 32) {
        const int p = base + lane;
        const uint32_t v = p < cf.HW ? (uint32_t)src[p] : 0u;
        uint32_t mine = 0;
        for (int c = 0; c < cf.C; ++c) {
            const uint32_t bits = __ballot_sync(0xffffffffu, (v >> c) & 1u);
            mine = lane == c ? bits : mine;
        }
        if (lane < cf.C)
            put_word(dbl, cf.NWP, lane, base >> 5, mine);
    }
}

// Six CTAs of eight warps per SM: 40 registers a thread (at 32 it spills and
// runs 6 % slower on the training shape).
template <typename CellT, int NA>
__global__ void __launch_bounds__(32 * kStepWarps, 6)
step_warp_kernel(DevConfig cf, const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
                 const uint32_t *__restrict__ vm_g, const uint32_t *__restrict__ masks_g, CellT *cur,
                 const CellT *__restrict__ init, int32_t *tsteps, const uint8_t *__restrict__ actions,
                 CellT *obs, int32_t *rew_out, uint8_t *done_out, int32_t *rew_sum, uint32_t *status)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const StepWarpLayout L = step_warp_layout(cf);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 3, q = lane & 7;
    const int NW = cf.NW, NWP = cf.NWP, C = cf.C, HW = cf.HW;
    uint32_t *vm = reinterpret_cast<uint32_t *>(smem + L.vm);
    uint32_t *masks = reinterpret_cast<uint32_t *>(smem + L.masks);
    for (int i = threadIdx.x; i < kShapes * NW; i += blockDim.x)
        vm[i] = __ldg(vm_g + i);
    for (int i = threadIdx.x; i < 3 * NW; i += blockDim.x)
        masks[i] = __ldg(masks_g + i);
    unsigned char *wr = smem + L.warps + (size_t)warp * L.per_warp;
    uint2 *planes = reinterpret_cast<uint2 *>(wr + L.planes);
    uint32_t *setp = reinterpret_cast<uint32_t *>(wr + L.setp);
    uint32_t *clrp = reinterpret_cast<uint32_t *>(wr + L.clrp);
    uint4 *hdr = reinterpret_cast<uint4 *>(wr + L.hdr);     // [R][2] the rule headers, copied
    uint2 *lead = reinterpret_cast<uint2 *>(wr + L.lead);  // [R][4 rotations][4] first term descriptors
    for (int i = lane; i < (C + 2) * NWP; i += 32)
        planes[i] = make_uint2(0u, 0u);
    for (int i = lane; i < C * NW; i += 32) {
        setp[i] = 0u;
        clrp[i] = 0u;
    }
    __syncthreads();  // the CTA's masks; no block barrier after this
    const int env = blockIdx.x * kStepWarps + warp;
    if (env >= cf.B)
        return;

    step_load_planes<CellT>(cf, cur + (size_t)env * HW, planes);
    int a = (int)actions[env];
    const bool warn = a > 4;
    if (warn)
        a = 0;
    __syncwarp();
    force_plane(cf, planes, masks, a);
    __syncwarp();

    // ---- every rule in its four rotations.  The headers, then every rule's
    // first four term descriptors, are copied in two passes, so that a rule
    // that fails its first four terms (most do) waits on no load from L2.
    const int table = cf.rules_per_env ? env : 0;
    const uint32_t *tab = arena + tab_off[table];
    const uint2 *terms = reinterpret_cast<const uint2 *>(tab + table_terms_word(cf.R));
    const uint2 pass = make_uint2((uint32_t)(C + 1) * NWP * 8, kTermAbsent);  // the zero plane, read as absent
    for (int i = lane; i < 2 * cf.R; i += 32)
        hdr[i] = __ldg(reinterpret_cast<const uint4 *>(tab + 4) + i);
    __syncwarp();
    for (int i = lane; i < 16 * cf.R; i += 32) {  // i = (rule, rotation, term)
        const int r = i >> 4, rot = (i >> 2) & 3, j = i & 3;
        const uint4 h0 = hdr[2 * r], h1 = hdr[2 * r + 1];
        lead[i] = (uint32_t)j < h0.x + h0.y ? __ldg(terms + (size_t)(h1.x + j) * 4 + rot) : pass;
    }
    __syncwarp();
    const uint4 *outs = reinterpret_cast<const uint4 *>(tab + table_outs_word(cf.R, __ldg(tab + 1)));
    const uint32_t pbase = (uint32_t)__cvta_generic_to_shared(planes) + q * 8;
    int rew = 0;
    for (int r = 0; r < cf.R; ++r) {
        const uint4 h0 = hdr[2 * r], h1 = hdr[2 * r + 1];
        const uint32_t *vmr = vm + ((h1.z >> (8 * g)) & 0xffu) * NW;
        uint32_t m[NA];
        uint32_t any = 0;
#pragma unroll
        for (int u = 0; u < NA; ++u) {
            const int w = q + 8 * u;
            m[u] = w < NW ? vmr[w] : 0u;
            any |= m[u];
        }
        const uint32_t nt = h0.x + h0.y;
        const uint2 *tp = terms + (size_t)h1.x * 4 + g;
        bool live = __any_sync(0xffffffffu, any != 0u);
        for (uint32_t t = 0; live && t < nt; t += 4) {
            uint2 d[4];
            if (t == 0) {  // the copied first four
                const uint4 *lp = reinterpret_cast<const uint4 *>(lead + (r * 4 + g) * 4);
                const uint4 x = lp[0], y = lp[1];
                d[0] = make_uint2(x.x, x.y);
                d[1] = make_uint2(x.z, x.w);
                d[2] = make_uint2(y.x, y.y);
                d[3] = make_uint2(y.z, y.w);
            } else {
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    d[j] = t + j < nt ? __ldg(tp + 4 * (t + j)) : pass;
            }
            any = 0;
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
        rew += (int)h0.w * (int)cnt;
        step_write<NA>(cf, outs + (size_t)h1.y * 4 + g, h0.z, m, setp, clrp);
    }
    rew = __reduce_add_sync(0xffffffffu, rew);

    // ---- combine: a bit changes where a match asks for it (SET on clear
    // cells, CLEAR on set cells); then the goal test, done and reset
    int goal = 0;
    for (int i = lane; i < C * NW; i += 32) {
        const int c = i / NW, w = i - c * NW;
        const uint32_t d = planes[c * NWP + w].x, st = setp[i], cl = clrp[i];
        const uint32_t nd = (d & ~cl) | (~d & st);
        if (nd != d)
            put_word(planes, NWP, c, w, nd);
        if (c == cf.ch_goal && nd)
            goal = 1;
    }
    const int goal_left = cf.ch_goal < 0 || __any_sync(0xffffffffu, goal);
    const int t = tsteps[env] + 1;
    const int done = !goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
    __syncwarp();
    if (done && cf.auto_reset)
        step_load_planes<CellT>(cf, init + (size_t)env * HW, planes);
    __syncwarp();
    step_store_cells<CellT>(cf, planes, cur + (size_t)env * HW, obs ? obs + (size_t)env * HW : nullptr);
    if (lane == 0) {
        tsteps[env] = done && cf.auto_reset ? 0 : t;
        if (rew_out)
            rew_out[env] = rew;
        if (done_out)
            done_out[env] = (uint8_t)done;
        if (rew_sum)
            rew_sum[env] = rew;
        if (warn)
            atomicOr(status + 1, kWarnAction);
    }
}

}  // namespace

cudaError_t configure_step()
{
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    };
    set((const void *)step_warp_kernel<uint8_t, 1>);
    set((const void *)step_warp_kernel<uint8_t, 2>);
    set((const void *)step_warp_kernel<uint16_t, 1>);
    set((const void *)step_warp_kernel<uint16_t, 2>);
    return e;
}

bool use_step_warp(const DevConfig &cf)
{
    return cf.path == 0 && cf.NA <= 2 && step_warp_layout(cf).total <= (size_t)kDynSmemLimit;
}

void launch_step_warp(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
                      const uint32_t *masks, void *cur, const void *init, int32_t *t, const uint8_t *actions,
                      void *obs, int32_t *rew, uint8_t *done, int32_t *rew_sum, uint32_t *status, cudaStream_t st)
{
    const size_t sm = step_warp_layout(cf).total;
    const int grid = (cf.B + kStepWarps - 1) / kStepWarps;
#define AV_STEP_LAUNCH(CELL, NA)                                                                            \
    step_warp_kernel<CELL, NA><<<grid, 32 * kStepWarps, sm, st>>>(                                          \
        cf, arena, tab_off, vm, masks, (CELL *)cur, (const CELL *)init, t, actions, (CELL *)obs, rew, done, \
        rew_sum, status)
    if (cf.cell_bytes == 1) {
        if (cf.NA == 1)
            AV_STEP_LAUNCH(uint8_t, 1);
        else
            AV_STEP_LAUNCH(uint8_t, 2);
    } else {
        if (cf.NA == 1)
            AV_STEP_LAUNCH(uint16_t, 1);
        else
            AV_STEP_LAUNCH(uint16_t, 2);
    }
#undef AV_STEP_LAUNCH
}

}  // namespace av
