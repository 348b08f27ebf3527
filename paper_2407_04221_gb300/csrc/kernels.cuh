// kernels.cuh -- device code of libautoverse.so (sm_103a).
//
// One CTA owns one environment (one board).  Each step:
//   A. board + force tile -> bit-planes in shared memory: plane c is the
//      board's channel-c bits as a row-major bit string of H*W bits, built
//      32 cells at a time with one warp ballot per channel.  Every plane word
//      j is stored doubled as (word j, word j+1) so that any 32-bit window of
//      the bit string is one 64-bit shared load plus one funnel shift.
//   B. matching (Sec. 2.1, ReLU(conv_{K_I}(D) - I + 1) == 1, evaluated as
//      bitwise AND): a work item is (rule rotation, anchor word a); its 32
//      bits are the anchors p = 32a + b.  Each term (channel c, window offset
//      s = i*W + k, present/absent) ANDs in bit p+s of plane c (or its
//      complement); the loop stops as soon as no anchor is left.  A match
//      pays the rule's reward and ORs the rule's output (set | clear << 16)
//      into a per-cell accumulator with shared-memory atomics: the
//      transposed-convolution write of Sec. 2.1.
//   C. combine next = (D & ~CLR) | (~D & SET) (force dropped), goal test by
//      a block-wide OR, reward by warp reductions.
//
// Rule table layout (uint32 words, one table per env or one shared table):
//   [0] K = 4R rule rotations   [1] n_items   [2] items_off   [3] terms_off
//   [4] outs_off (even)          [5..7] 0
//   [8 + 8*rr ...] header of rotation rr: shape = (h'-1)*5 + (w'-1),
//        n_terms, n_outs, reward, first term, first out, 0, 0
//   items:  (rr << 16) | a, every anchor word that holds a valid anchor
//   terms:  (byte offset of plane c, word s>>5) << 8 | absent << 5 | (s & 31)
//   outs:   pairs (cell offset i*W + k, set | clear << 16)
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace av {

constexpr int kThreads = 256;
constexpr int kPlanePad = 10;     // doubled-plane entries past the last word
constexpr int kMaxCand = 4096;    // av_select: candidates per env
constexpr uint32_t kStatusVisitedOverflow = 1u;
constexpr uint32_t kWarnAction = 1u;

struct DevConfig {
    int B, H, W, C, HW, NW, NWP, pstride;
    int R, rules_per_env, max_steps, auto_reset;
    int ch_player, ch_goal, ch_empty, ch_wall, border_wall, cum_per_env;
    int cell_bytes;
};

__host__ __device__ inline uint32_t encode_term(int c, int s, int neg, int pstride)
{
    return ((uint32_t)(c * pstride + (s >> 5) * 8) << 8) | ((uint32_t)neg << 5) | (uint32_t)(s & 31);
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
    size_t planes, sc, boards, red, total;
};

// Layout: planes | SC accumulators | n_boards boards of uint16 cells | 3 reward slots
__host__ __device__ inline StepSmem step_smem(const DevConfig &cf, int n_boards)
{
    StepSmem s;
    s.planes = 0;
    s.sc = align16((size_t)(cf.C + 1) * cf.NWP * 8);
    s.boards = align16(s.sc + (size_t)cf.HW * 4);
    s.red = align16(s.boards + (size_t)cf.HW * 2 * n_boards);
    s.total = s.red + 16;
    return s;
}

struct StepOut {
    int reward;
    int goal_left;
};

// One transition of the board in `gin` into `gout` (both shared, uint16 cells).
// `slot` is a zeroed shared int used for the block's reward sum.
__device__ StepOut step_body(const DevConfig &cf, const uint32_t *__restrict__ tab,
                             const uint32_t *__restrict__ vm, uint2 *planes, uint32_t *SC,
                             const uint16_t *gin, uint16_t *gout, int action, int *slot)
{
    const int tid = threadIdx.x, lane = tid & 31;
    const int HW = cf.HW, H = cf.H, W = cf.W, C = cf.C, NCH = C + 1, NWP = cf.NWP;

    // ---- A: board + force -> bit-planes
    int dy = 0, dx = 0;
    if (cf.ch_player >= 0) {
        if (action == 1) dy = -1;
        else if (action == 2) dx = 1;
        else if (action == 3) dy = 1;
        else if (action == 4) dx = -1;
    }
    const bool force = (dy | dx) != 0;
    for (int base = 0; base < HW; base += blockDim.x) {
        const int p = base + tid;
        uint32_t v = 0;
        if (p < HW) {
            v = gin[p];
            if (force) {
                const int y = p / W, x = p - y * W;
                const int sy = y - dy, sx = x - dx;
                if ((unsigned)sy < (unsigned)H && (unsigned)sx < (unsigned)W &&
                    ((gin[sy * W + sx] >> cf.ch_player) & 1u))
                    v |= 1u << C;
            }
        }
        const int w = p >> 5;
        for (int c = 0; c < NCH; ++c) {
            const uint32_t bits = __ballot_sync(0xffffffffu, (v >> c) & 1u);
            if (lane == 0 && w < cf.NW) {
                planes[c * NWP + w].x = bits;
                if (w > 0)
                    planes[c * NWP + w - 1].y = bits;
            }
        }
    }
    __syncthreads();

    // ---- B: match every (rule rotation, anchor word) item
    const uint32_t n_items = tab[1];
    const uint32_t *items = tab + tab[2];
    const uint32_t *terms = tab + tab[3];
    const uint2 *outs = reinterpret_cast<const uint2 *>(tab + tab[4]);
    const uint32_t *hdr = tab + 8;
    const char *pbase = reinterpret_cast<const char *>(planes);
    int rew = 0;
    for (uint32_t it = tid; it < n_items; it += blockDim.x) {
        const uint32_t item = __ldg(items + it);
        const uint32_t rr = item >> 16, a = item & 0xffffu;
        const uint4 h0 = __ldg(reinterpret_cast<const uint4 *>(hdr + 8 * rr));
        const uint2 h1 = __ldg(reinterpret_cast<const uint2 *>(hdr + 8 * rr + 4));
        uint32_t m = __ldg(vm + h0.x * cf.NW + a);
        const char *abase = pbase + a * 8;
        const uint32_t *tp = terms + h1.x;
        for (uint32_t t = 0; t < h0.y && m; ++t) {
            const uint32_t e = __ldg(tp + t);
            const uint2 wd = *reinterpret_cast<const uint2 *>(abase + (e >> 8));
            const uint32_t x = __funnelshift_r(wd.x, wd.y, e & 31u);
            m &= (e & 32u) ? ~x : x;
        }
        if (m) {
            rew += (int)h0.w * __popc(m);
            const uint2 *op = outs + h1.y;
            uint32_t mm = m;
            while (mm) {
                const int b = __ffs(mm) - 1;
                mm &= mm - 1;
                const int p = (int)a * 32 + b;
                for (uint32_t o = 0; o < h0.z; ++o) {
                    const uint2 ov = __ldg(op + o);
                    atomicOr(&SC[p + (int)ov.x], ov.y);
                }
            }
        }
    }
    rew = __reduce_add_sync(0xffffffffu, rew);
    if (lane == 0 && rew)
        atomicAdd(slot, rew);
    __syncthreads();

    // ---- C: combine, goal test
    const uint32_t tiles = (1u << C) - 1u;
    int any_goal = 0;
    for (int p = tid; p < HW; p += blockDim.x) {
        const uint32_t v = gin[p];
        const uint32_t sc = SC[p];
        if (sc)
            SC[p] = 0;
        const uint32_t set = sc & 0xffffu, clr = sc >> 16;
        const uint32_t nv = ((v & ~clr) | (~v & set)) & tiles;
        gout[p] = (uint16_t)nv;
        if (cf.ch_goal >= 0)
            any_goal |= (int)((nv >> cf.ch_goal) & 1u);
    }
    StepOut o;
    o.goal_left = __syncthreads_or(any_goal);
    if (cf.ch_goal < 0)
        o.goal_left = 1;
    o.reward = *slot;
    return o;
}

// ---------------------------------------------------------------- kernels
template <typename CellT>
__global__ void __launch_bounds__(kThreads)
rollout_kernel(DevConfig cf, const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
               const uint32_t *__restrict__ vm, CellT *cur, const CellT *__restrict__ init,
               int32_t *tsteps, int n_steps, uint64_t seed, const uint8_t *__restrict__ actions,
               CellT *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
               uint32_t *status)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const StepSmem L = step_smem(cf, 3);
    const int env = blockIdx.x, tid = threadIdx.x, HW = cf.HW;
    uint2 *planes = reinterpret_cast<uint2 *>(smem + L.planes);
    uint32_t *SC = reinterpret_cast<uint32_t *>(smem + L.sc);
    uint16_t *G0 = reinterpret_cast<uint16_t *>(smem + L.boards);
    uint16_t *G1 = G0 + HW, *GI = G1 + HW;
    int *red = reinterpret_cast<int *>(smem + L.red);
    const uint32_t *tab = arena + tab_off[cf.rules_per_env ? env : 0];

    for (int i = tid; i < (cf.C + 1) * cf.NWP; i += blockDim.x)
        planes[i] = make_uint2(0u, 0u);
    const CellT *src = cur + (size_t)env * HW;
    const CellT *isrc = init + (size_t)env * HW;
    for (int p = tid; p < HW; p += blockDim.x) {
        SC[p] = 0;
        G0[p] = (uint16_t)src[p];
        GI[p] = (uint16_t)isrc[p];
    }
    if (tid < 3)
        red[tid] = 0;
    __syncthreads();

    int t = tsteps[env];
    int sum = 0;
    uint32_t warn = 0;
    uint16_t *gin = G0, *gout = G1;
    for (int s = 0; s < n_steps; ++s) {
        int a = actions ? (int)actions[env] : (int)uniform_below(draw(seed, 4, (uint64_t)env, 0, (uint64_t)s), 5);
        if (a > 4) {
            warn = kWarnAction;
            a = 0;
        }
        if (tid == 0)
            red[(s + 1) % 3] = 0;
        const StepOut o = step_body(cf, tab, vm, planes, SC, gin, gout, a, &red[s % 3]);
        t += 1;
        const int done = !o.goal_left || (cf.max_steps > 0 && t >= cf.max_steps);
        if (done && cf.auto_reset) {
            for (int p = tid; p < HW; p += blockDim.x)
                gout[p] = GI[p];
            t = 0;
            __syncthreads();
        }
        if (obs_traj) {
            CellT *dst = obs_traj + ((size_t)s * cf.B + env) * HW;
            for (int p = tid; p < HW; p += blockDim.x)
                dst[p] = (CellT)gout[p];
        }
        if (tid == 0) {
            if (rew_traj)
                rew_traj[(size_t)s * cf.B + env] = o.reward;
            if (done_traj)
                done_traj[(size_t)s * cf.B + env] = (uint8_t)done;
        }
        sum += o.reward;
        uint16_t *tmp = gin;
        gin = gout;
        gout = tmp;
    }
    CellT *dst = cur + (size_t)env * HW;
    for (int p = tid; p < HW; p += blockDim.x)
        dst[p] = (CellT)gin[p];
    if (tid == 0) {
        tsteps[env] = t;
        if (rew_sum)
            rew_sum[env] = sum;
        if (warn)
            atomicOr(status + 1, warn);
    }
}

template <typename CellT>
__global__ void __launch_bounds__(kThreads)
expand_kernel(DevConfig cf, const uint32_t *__restrict__ arena, const uint32_t *__restrict__ tab_off,
              const uint32_t *__restrict__ vm, const CellT *__restrict__ parents, int F,
              const int32_t *__restrict__ n_parent, CellT *children, int32_t *rewards,
              uint8_t *done, uint64_t *hashes)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const StepSmem L = step_smem(cf, 6);
    const int node = blockIdx.x, env = node / F, tid = threadIdx.x, HW = cf.HW;
    if (n_parent && node - env * F >= n_parent[env])
        return;  // block-uniform: an empty frontier slot
    uint2 *planes = reinterpret_cast<uint2 *>(smem + L.planes);
    uint32_t *SC = reinterpret_cast<uint32_t *>(smem + L.sc);
    uint16_t *G0 = reinterpret_cast<uint16_t *>(smem + L.boards);
    int *red = reinterpret_cast<int *>(smem + L.red);
    const uint32_t *tab = arena + tab_off[cf.rules_per_env ? env : 0];

    for (int i = tid; i < (cf.C + 1) * cf.NWP; i += blockDim.x)
        planes[i] = make_uint2(0u, 0u);
    const CellT *src = parents + (size_t)node * HW;
    for (int p = tid; p < HW; p += blockDim.x) {
        SC[p] = 0;
        G0[p] = (uint16_t)src[p];
    }
    if (tid < 3)
        red[tid] = 0;
    __syncthreads();

    for (int a = 0; a < 5; ++a) {
        uint16_t *gc = G0 + (size_t)(a + 1) * HW;
        if (tid == 0)
            red[(a + 1) % 3] = 0;
        const StepOut o = step_body(cf, tab, vm, planes, SC, G0, gc, a, &red[a % 3]);
        const size_t slot = (size_t)node * 5 + a;
        CellT *dst = children + slot * HW;
        for (int p = tid; p < HW; p += blockDim.x)
            dst[p] = (CellT)gc[p];
        if (tid == 0) {
            rewards[slot] = o.reward;
            if (done)
                done[slot] = (uint8_t)!o.goal_left;
        }
    }
    // children are complete: every step ended with a block-wide barrier.
    // FNV-1a 64 over the canonical bytes, one thread per child.
    if ((tid & 31) == 0 && (tid >> 5) < 5) {
        const int a = tid >> 5;
        const uint16_t *gc = G0 + (size_t)(a + 1) * HW;
        uint64_t hsh = 0xcbf29ce484222325ULL;
        for (int p = 0; p < HW; ++p) {
            const uint32_t v = gc[p];
            hsh = (hsh ^ (v & 0xffu)) * 0x100000001b3ULL;
            if (sizeof(CellT) == 2)
                hsh = (hsh ^ (v >> 8)) * 0x100000001b3ULL;
        }
        hashes[(size_t)node * 5 + a] = hsh;
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
template <typename CellT>
__global__ void search_init_kernel(DevConfig cf, int cap, const CellT *__restrict__ roots,
                                   uint64_t *root_hash, uint8_t *root_live, uint64_t *visited,
                                   int32_t *n_visited)
{
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
    visited[(size_t)b * cap] = hsh;  // parity 0
    n_visited[b] = 1;
}

struct Key128 {
    uint64_t hi, lo;
};

__device__ __forceinline__ bool key_less(const Key128 &a, const Key128 &b)
{
    return a.hi < b.hi || (a.hi == b.hi && a.lo < b.lo);
}

// Block-wide bitonic sort of n2 (power of two) keys in shared memory, ascending.
__device__ void bitonic_sort(Key128 *keys, int n2)
{
    for (int k = 2; k <= n2; k <<= 1)
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = threadIdx.x; i < n2; i += blockDim.x) {
                const int ixj = i ^ j;
                if (ixj > i) {
                    const bool up = (i & k) == 0;
                    Key128 x = keys[i], y = keys[ixj];
                    if (key_less(y, x) == up) {
                        keys[i] = y;
                        keys[ixj] = x;
                    }
                }
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
        for (int i = tid; i < nv; i += blockDim.x)
            vis_out[i] = vis_in[i];
        return;
    }
    for (int i = tid; i < nv; i += blockDim.x)
        vis_out[i + lower_bound_u64(sel, take, vis_in[i])] = vis_in[i];
    for (int j = tid; j < take; j += blockDim.x)
        vis_out[j + lower_bound_u64(vis_in, nv, sel[j])] = sel[j];
    if (tid == 0)
        n_visited[b] = nv + take;
}

// ------------------------------------------------------------ launchers
inline size_t select_smem_bytes(int F)
{
    int n2 = 1;
    while (n2 < 5 * F)
        n2 <<= 1;
    // sort keys (n2) + selected hashes (n2 uint64) + their sort keys (n2)
    return (size_t)n2 * sizeof(Key128) * 2 + (size_t)n2 * 8 + 64;
}

inline cudaError_t configure_kernels(const DevConfig &cf)
{
    const int big = 200 * 1024;
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, big);
    };
    if (cf.cell_bytes == 1) {
        set((const void *)rollout_kernel<uint8_t>);
        set((const void *)expand_kernel<uint8_t>);
        set((const void *)reset_kernel<uint8_t>);
        set((const void *)select_kernel<uint8_t>);
        set((const void *)search_init_kernel<uint8_t>);
    } else {
        set((const void *)rollout_kernel<uint16_t>);
        set((const void *)expand_kernel<uint16_t>);
        set((const void *)reset_kernel<uint16_t>);
        set((const void *)select_kernel<uint16_t>);
        set((const void *)search_init_kernel<uint16_t>);
    }
    return e;
}

inline void launch_rollout(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                           const uint32_t *vm, void *cur, const void *init, int32_t *t, int n_steps,
                           uint64_t seed, const uint8_t *actions, void *obs_traj, int32_t *rew_traj,
                           uint8_t *done_traj, int32_t *rew_sum, uint32_t *status, cudaStream_t st)
{
    const size_t sm = step_smem(cf, 3).total;
    if (cf.cell_bytes == 1)
        rollout_kernel<uint8_t><<<cf.B, kThreads, sm, st>>>(
            cf, arena, tab_off, vm, (uint8_t *)cur, (const uint8_t *)init, t, n_steps, seed, actions,
            (uint8_t *)obs_traj, rew_traj, done_traj, rew_sum, status);
    else
        rollout_kernel<uint16_t><<<cf.B, kThreads, sm, st>>>(
            cf, arena, tab_off, vm, (uint16_t *)cur, (const uint16_t *)init, t, n_steps, seed, actions,
            (uint16_t *)obs_traj, rew_traj, done_traj, rew_sum, status);
}

inline void launch_expand(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                          const uint32_t *vm, const void *parents, int F, const int32_t *n_parent,
                          void *children, int32_t *rewards, uint8_t *done, uint64_t *hashes,
                          cudaStream_t st)
{
    const size_t sm = step_smem(cf, 6).total;
    const unsigned grid = (unsigned)(cf.B * F);
    if (cf.cell_bytes == 1)
        expand_kernel<uint8_t><<<grid, kThreads, sm, st>>>(cf, arena, tab_off, vm, (const uint8_t *)parents,
                                                          F, n_parent, (uint8_t *)children, rewards, done,
                                                          hashes);
    else
        expand_kernel<uint16_t><<<grid, kThreads, sm, st>>>(cf, arena, tab_off, vm, (const uint16_t *)parents,
                                                           F, n_parent, (uint16_t *)children, rewards, done,
                                                           hashes);
}

inline void launch_reset(const DevConfig &cf, const uint32_t *cum, uint64_t seed, void *cur, void *init,
                         int32_t *t, void *obs, cudaStream_t st)
{
    const size_t sm = align16((size_t)cf.HW * 2);
    if (cf.cell_bytes == 1)
        reset_kernel<uint8_t><<<cf.B, kThreads, sm, st>>>(cf, cum, seed, (uint8_t *)cur, (uint8_t *)init, t,
                                                         (uint8_t *)obs);
    else
        reset_kernel<uint16_t><<<cf.B, kThreads, sm, st>>>(cf, cum, seed, (uint16_t *)cur, (uint16_t *)init,
                                                          t, (uint16_t *)obs);
}

inline void launch_search_init(const DevConfig &cf, int cap, const void *roots, uint64_t *root_hash,
                               uint8_t *root_live, uint64_t *visited, int32_t *n_visited, cudaStream_t st)
{
    const unsigned grid = (unsigned)((cf.B + 127) / 128);
    if (cf.cell_bytes == 1)
        search_init_kernel<uint8_t><<<grid, 128, 0, st>>>(cf, cap, (const uint8_t *)roots, root_hash, root_live,
                                                         visited, n_visited);
    else
        search_init_kernel<uint16_t><<<grid, 128, 0, st>>>(cf, cap, (const uint16_t *)roots, root_hash,
                                                          root_live, visited, n_visited);
}

inline void launch_select(const DevConfig &cf, int cap, int parity, int F, const int32_t *n_parent,
                          const int32_t *parent_cum, const uint8_t *parent_live, const void *cand_grids,
                          const int32_t *cand_reward, const uint8_t *cand_done, const uint64_t *cand_hash,
                          int k, void *next_grids, int32_t *next_cum, uint64_t *next_hash,
                          uint8_t *next_live, int32_t *n_next, uint64_t *visited, int32_t *n_visited,
                          uint32_t *status, cudaStream_t st)
{
    const size_t sm = select_smem_bytes(F);
    if (cf.cell_bytes == 1)
        select_kernel<uint8_t><<<cf.B, kThreads, sm, st>>>(
            cf, cap, parity, F, n_parent, parent_cum, parent_live, (const uint8_t *)cand_grids, cand_reward,
            cand_done, cand_hash, k, (uint8_t *)next_grids, next_cum, next_hash, next_live, n_next, visited,
            n_visited, status);
    else
        select_kernel<uint16_t><<<cf.B, kThreads, sm, st>>>(
            cf, cap, parity, F, n_parent, parent_cum, parent_live, (const uint16_t *)cand_grids, cand_reward,
            cand_done, cand_hash, k, (uint16_t *)next_grids, next_cum, next_hash, next_live, n_next, visited,
            n_visited, status);
}

}  // namespace av
