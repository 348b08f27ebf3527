// k_mutate.cu -- the mutation operators of the evolution loop (Sec. 3.1.1):
// bits of the initial maps flipped at random, tiles of the mutable rules'
// input and output patterns changed, rule rewards redrawn.  Every decision
// is one counter draw,
//     draw(seed, st, a, b, c) = mix(mix(mix(seed + golden*(st+1)) ^ a) ^ (b<<32 | c)),
// taken when its top 24 bits are below the rate (in units of 2^-24):
//   map bit (cell q, channel c) of env b:      st 9,  a = b, b = q,          c = c
//   input entry (rule r, entry e, channel c):   st 10, a = t, b = 25 r + e,   c = c
//   output entry (rule r, entry e, channel c):  st 11, a = t, b = 25 r + e,   c = c
//   reward of rule r:                           st 12, a = t, b = r, c = 0 (decision), 1 (value)
// A changed ternary entry moves to the next state (cyclically) when bit 39 of
// its draw is 0, to the one after when 1.
//
// One warp per environment (map) or rule table: the first two mixes depend
// only on (seed, stream, environment), so each lane computes them once and
// then one mix per decision.  Rule entries are dealt to lanes from a dense
// list of the table's existing (rule, entry) pairs.
#include <algorithm>

#include "launch.h"

namespace av {
namespace {

constexpr int kMutThreads = 256;

// mix(mix(seed + golden*(st+1)) ^ a): the part of draw() shared by every
// decision of one environment in one stream.
__device__ __forceinline__ uint64_t draw_prefix(uint64_t seed, uint64_t st, uint64_t a)
{
    return mix64(mix64(seed + 0x9E3779B97F4A7C15ULL * (st + 1)) ^ a);
}

__device__ __forceinline__ uint64_t draw_from(uint64_t prefix, uint64_t b, uint64_t c)
{
    return mix64(prefix ^ ((b << 32) | c));
}

template <typename CellT>
__global__ void __launch_bounds__(kMutThreads)
    mutate_maps_kernel(int B, int HW, int C, uint32_t p_map, uint32_t channels, uint64_t seed, CellT *maps)
{
    const int lane = threadIdx.x & 31;
    const int warps = gridDim.x * (kMutThreads / 32);
    for (int b = blockIdx.x * (kMutThreads / 32) + (threadIdx.x >> 5); b < B; b += warps) {
        const uint64_t pre = draw_prefix(seed, 9, (uint64_t)b);
        CellT *m = maps + (size_t)b * HW;
        for (int q = lane; q < HW; q += 32) {
            uint32_t flip = 0;
            for (int c = 0; c < C; ++c)
                if (((channels >> c) & 1u) && (uint32_t)(draw_from(pre, (uint64_t)q, (uint64_t)c) >> 40) < p_map)
                    flip |= 1u << c;
            if (flip)
                m[q] = (CellT)(m[q] ^ flip);
        }
    }
}

// Packed record as 32-bit words: [0] h | w << 8, [1] reward, [2 + e] present,
// [27 + e] absent, [52 + e] set, [77 + e] clear.
constexpr int kRecWords = 102;

// New ternary state of bit c of the mask pair (one, two) after decision d.
__device__ __forceinline__ void mutate_entry(uint32_t &one, uint32_t &two, int c, uint64_t d, uint32_t p)
{
    if ((uint32_t)(d >> 40) >= p)
        return;
    const uint32_t bit = 1u << c;
    const int state = (one & bit) ? 1 : (two & bit) ? 2 : 0;
    const int next = (state + 1 + (int)((d >> 39) & 1u)) % 3;
    one &= ~bit;
    two &= ~bit;
    if (next == 1)
        one |= bit;
    else if (next == 2)
        two |= bit;
}

__global__ void __launch_bounds__(kMutThreads)
    mutate_rules_kernel(int T, int R, int C, uint32_t p_rule, uint32_t p_reward, int32_t reward_min,
                        uint64_t reward_span, uint64_t mutable_rules, uint64_t seed, uint32_t *rules)
{
    // Per warp: offsets of each rule's entries in the dense list of the
    // table's mutable (rule, pattern entry) pairs, so that lanes stride over
    // entries that exist (a 1 x 2 pattern has 2 of the 25 slots).
    __shared__ int s_off[kMutThreads / 32][2 * 32 + 1];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    int *off = s_off[wid];
    const int warps = gridDim.x * (kMutThreads / 32);
    for (int t = blockIdx.x * (kMutThreads / 32) + wid; t < T; t += warps) {
        uint32_t *tab = rules + (size_t)t * R * kRecWords;
        if (p_rule > 0) {
            int total = 0;
            for (int half = 0; half < 2; ++half) {  // rules lane and lane + 32
                const int r = lane + 32 * half;
                int n = 0;
                if (r < R && ((mutable_rules >> r) & 1u)) {
                    const uint32_t hw = tab[(size_t)r * kRecWords];
                    n = min(25, (int)(hw & 0xffu) * (int)((hw >> 8) & 0xffu));  // 25 entries per record
                }
                for (int d = 1; d < 32; d <<= 1) {  // inclusive scan
                    const int v = __shfl_up_sync(0xffffffffu, n, d);
                    if (lane >= d)
                        n += v;
                }
                off[1 + 32 * half + lane] = total + n;
                total += __shfl_sync(0xffffffffu, n, 31);
            }
            if (lane == 0)
                off[0] = 0;
            __syncwarp();
            const uint64_t pre_in = draw_prefix(seed, 10, (uint64_t)t);
            const uint64_t pre_out = draw_prefix(seed, 11, (uint64_t)t);
            for (int j = lane; j < total; j += 32) {
                int lo = 0, hi = 64;  // the rule r with off[r] <= j < off[r + 1]
                while (hi - lo > 1) {
                    const int mid = (lo + hi) >> 1;
                    if (off[mid] <= j)
                        lo = mid;
                    else
                        hi = mid;
                }
                const int r = lo, e = j - off[r];
                const uint64_t k = (uint64_t)(25 * r + e);
                uint32_t *rec = tab + (size_t)r * kRecWords;
                uint32_t pres = rec[2 + e], absn = rec[27 + e], set = rec[52 + e], clr = rec[77 + e];
                for (int c = 0; c <= C; ++c)
                    mutate_entry(pres, absn, c, draw_from(pre_in, k, (uint64_t)c), p_rule);
                for (int c = 0; c < C; ++c)
                    mutate_entry(set, clr, c, draw_from(pre_out, k, (uint64_t)c), p_rule);
                rec[2 + e] = pres;
                rec[27 + e] = absn;
                rec[52 + e] = set;
                rec[77 + e] = clr;
            }
            __syncwarp();  // off[] is rewritten for the next table
        }
        if (p_reward > 0) {
            const uint64_t pre_rw = draw_prefix(seed, 12, (uint64_t)t);
            for (int r = lane; r < R; r += 32) {
                if (!((mutable_rules >> r) & 1u))
                    continue;
                if ((uint32_t)(draw_from(pre_rw, (uint64_t)r, 0) >> 40) < p_reward) {
                    const uint64_t u = draw_from(pre_rw, (uint64_t)r, 1) >> 32;
                    tab[(size_t)r * kRecWords + 1] = (uint32_t)(reward_min + (int64_t)((u * reward_span) >> 32));
                }
            }
        }
    }
}

int mutate_grid(int n_warp_units)
{
    const int per_cta = kMutThreads / 32;
    return std::max(1, std::min((n_warp_units + per_cta - 1) / per_cta, 152 * 8));
}

}  // namespace

void launch_mutate(int B, int H, int W, int C, int R, uint32_t p_map, uint32_t map_channels, uint32_t p_rule,
                   uint32_t p_reward, int32_t reward_min, int32_t reward_max, uint64_t mutable_rules, uint64_t seed,
                   void *maps, uint32_t *rules, cudaStream_t st)
{
    const uint32_t channels = map_channels & ((1u << C) - 1u);
    if (maps != nullptr && p_map > 0 && channels != 0) {
        if (C <= 8)
            mutate_maps_kernel<uint8_t><<<mutate_grid(B), kMutThreads, 0, st>>>(B, H * W, C, p_map, channels, seed,
                                                                                 (uint8_t *)maps);
        else
            mutate_maps_kernel<uint16_t><<<mutate_grid(B), kMutThreads, 0, st>>>(B, H * W, C, p_map, channels, seed,
                                                                                  (uint16_t *)maps);
    }
    const uint64_t mask = R >= 64 ? ~0ull : ((1ull << R) - 1ull);
    if (rules != nullptr && R > 0 && (mutable_rules & mask) != 0 && (p_rule > 0 || p_reward > 0)) {
        const uint64_t span = (uint64_t)((int64_t)reward_max - (int64_t)reward_min + 1);
        mutate_rules_kernel<<<mutate_grid(B), kMutThreads, 0, st>>>(B, R, C, p_rule, p_reward, reward_min, span,
                                                                   mutable_rules, seed, rules);
    }
}

}  // namespace av
