// k_observe.cu -- the policy observation (Sec. 3.2, imitation learning: the
// agent sees a local patch of tiles centred on the player plus a binary form
// of the environment's rules; Sec. 4, Tables 1 and 2: patch widths 5 to 31,
// zero padding outside the map, hidden rules as zeros).
//
// observe_kernel: a persistent kernel over groups of consecutive
// environments (one environment per group for large patches, up to eight for
// small ones; their boards and patches are contiguous).  A group's boards are
// fetched into shared memory with cp.async while the previous group's patches
// are built (boards over 8 KB, up to 256 x 256, are read from global memory
// instead); each environment's player is its first row-major cell with the
// player bit (a warp reduction, then an atomicMin).  The patches -- [window]
// [window][C] bytes each, channels last -- are built in a staging slab that is
// zero-filled with 16-byte stores, after which only the set tile bits of the
// board cells inside each window are written (a cell holds one or two of its
// C channels, so most bytes are zeros).  The slab's 16-byte-aligned middle
// leaves by one bulk TMA store (cp.async.bulk, shared to global) that the CTA
// does not wait for until the slab is needed again; the unaligned head and
// tail bytes are plain stores, so every output byte is written by exactly one
// CTA whatever the alignment.  Patches larger than the slab go out in row
// slabs.
//
// rule_obs_kernel: one thread per (rule, plane, frame entry) writes the C + 1
// channel bytes of that entry from the packed 408-byte record.
#include <algorithm>

#include "launch.h"

namespace av {
namespace {

constexpr int kObsThreads = 128;
constexpr int kObsSlabBytes = 32768;  // patch bytes staged per slab

__device__ __forceinline__ uint32_t shared_addr(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

// Bulk copy of `bytes` (a multiple of 16) from shared to global memory by the
// TMA unit; both addresses 16-byte aligned.
__device__ __forceinline__ void bulk_store(void *gdst, const void *ssrc, uint32_t bytes)
{
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;"
                 :
                 : "l"(gdst), "r"(shared_addr(ssrc)), "r"(bytes)
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

// Wait until at most N of the issued bulk-store groups have still to read
// their shared source.
template <int N>
__device__ __forceinline__ void bulk_wait_read()
{
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}

// Make this thread's ordinary shared-memory writes visible to the TMA unit.
__device__ __forceinline__ void fence_async_shared() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// 16-byte asynchronous copy global -> shared (both 16-byte aligned).
__device__ __forceinline__ void cp_async16(void *sdst, const void *gsrc)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(shared_addr(sdst)), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// Start copying HW cells (one or more boards) into shared memory:
// asynchronous 16-byte copies when the bytes allow (vec16), else plain loads.
template <typename CellT>
__device__ __forceinline__ void fetch_board(CellT *dst, const CellT *src, int HW, int vec16)
{
    if (vec16) {  // HW * sizeof(CellT) is a multiple of 16
        const int n16 = (int)((size_t)HW * sizeof(CellT) / 16);
        for (int j = threadIdx.x; j < n16; j += kObsThreads)
            cp_async16(reinterpret_cast<uint4 *>(dst) + j, reinterpret_cast<const uint4 *>(src) + j);
    } else {
        for (int q = threadIdx.x; q < HW; q += kObsThreads)
            dst[q] = src[q];
    }
    cp_async_commit();
}

constexpr int kObsGroupMax = 8;  // environments per group (small patches)

// Persistent: CTA c observes groups c, c + gridDim.x, ... of E consecutive
// environments (E > 1 for small patches, so that one board fetch and one bulk
// store serve E patches: boards and patches of consecutive environments are
// contiguous).  Two board buffers and two staging slabs form a pipeline: the
// next group's boards are fetched while the current patches are built, and a
// slab is rewritten only after the bulk store issued from it two units
// earlier has read it.  A unit is one slab: a whole group's patches, or, for
// a patch larger than kObsSlabBytes (E = 1), a range of its rows.
template <typename CellT>
__global__ void __launch_bounds__(kObsThreads)
    observe_kernel(int B, int H, int W, int C, int ch_player, const CellT *__restrict__ grids, int window,
                   uint8_t *__restrict__ obs, int32_t *__restrict__ player_yx, int E, int rows_per_slab,
                   int board_region, int buf_region, int vec16)
{
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ int s_first[2][kObsGroupMax];
    const int HW = H * W;
    const int tid = threadIdx.x;
    const int n_groups = (B + E - 1) / E;
    int g = blockIdx.x;
    if (g >= n_groups)
        return;
    // Shared memory: boards 0, boards 1, slab 0, slab 1.
    auto board_at = [&](int i) { return reinterpret_cast<CellT *>(smem + i * board_region); };
    auto slab_at = [&](uint32_t i) { return smem + 2 * board_region + (int)(i & 1u) * buf_region; };
    const size_t row_bytes = (size_t)window * C;
    const size_t patch_bytes = row_bytes * window;
    const uint32_t tile_bits = (1u << C) - 1u;  // bits >= C of a caller's board are not tiles
    // Teams of threads per patch: the whole CTA for one patch per group, half
    // of it for two, one warp for four or more.
    const int team = E == 1 ? kObsThreads : E == 2 ? kObsThreads / 2 : 32;
    const int n_teams = kObsThreads / team;
    const int my_team = tid / team, team_tid = tid % team;
    auto group_size = [&](int grp) { return min(E, B - grp * E); };
    if (tid < E)
        s_first[0][tid] = HW;
    if (board_region)  // else boards are read from global memory where they lie
        fetch_board(board_at(0), grids + (size_t)g * E * HW, group_size(g) * HW, vec16);
    uint32_t unit = 0;  // slabs issued so far; slab buffer = unit & 1
    for (int it = 0; g < n_groups; ++it, g += gridDim.x) {
        const int pb = it & 1;
        const int ne = group_size(g);
        const CellT *board = board_region ? board_at(pb) : grids + (size_t)g * E * HW;
        uint8_t *out = obs + (size_t)g * E * patch_bytes;
        if (tid == 0)
            bulk_wait_read<1>();  // slab_at(unit) has been read by its last store
        cp_async_wait_all();
        __syncthreads();  // the group's boards in shared memory; s_first[pb] reset; slab free
        const int gn = g + gridDim.x;
        if (board_region && gn < n_groups)
            fetch_board(board_at(pb ^ 1), grids + (size_t)gn * E * HW, group_size(gn) * HW, vec16);
        // Each environment's player: its first row-major cell holding the
        // player bit.  A thread's first hit is its minimum; a warp reduces its
        // lanes' hits and makes one atomicMin.
        for (int e = my_team; e < ne; e += n_teams) {
            int hit = HW;
            for (int q = team_tid; q < HW; q += team)
                if ((board[e * HW + q] >> ch_player) & 1) {
                    hit = q;
                    break;
                }
            hit = __reduce_min_sync(0xffffffffu, hit);
            if ((tid & 31) == 0 && hit < HW)
                atomicMin(&s_first[pb][e], hit);
        }
        const size_t group_bytes = (size_t)ne * patch_bytes;
        const int slab_rows = E == 1 ? rows_per_slab : window;
        for (int r0 = 0; r0 < window; r0 += slab_rows, ++unit) {
            const int r1 = min(window, r0 + slab_rows);
            uint8_t *gs = out + (size_t)r0 * row_bytes;
            uint8_t *buf = slab_at(unit);
            const uint32_t len = (uint32_t)(E == 1 ? (size_t)(r1 - r0) * row_bytes : group_bytes);
            const uint32_t shift = (uint32_t)(reinterpret_cast<uintptr_t>(gs) & 15u);  // buf[shift] <-> gs[0]
            if (r0 > 0) {  // a further slab of this patch: wait for its buffer
                if (tid == 0)
                    bulk_wait_read<1>();
                __syncthreads();
            }
            const uint32_t words = (shift + len + 15u) >> 4;
            uint4 *buf4 = reinterpret_cast<uint4 *>(buf);
            for (uint32_t j = tid; j < words; j += kObsThreads)
                buf4[j] = make_uint4(0u, 0u, 0u, 0u);
            __syncthreads();  // slab zeroed; players known
            for (int e = my_team; e < ne; e += n_teams) {
                const int first = s_first[pb][e];
                const bool has_player = first < HW;
                const int py = has_player ? first / W : -1;
                const int px = has_player ? first - py * W : -1;
                if (r0 == 0 && team_tid == 0 && player_yx != nullptr) {
                    player_yx[2 * ((size_t)g * E + e)] = py;
                    player_yx[2 * ((size_t)g * E + e) + 1] = px;
                }
                const int y0 = py - window / 2, x0 = px - window / 2;  // board cell of patch entry (0, 0)
                const int xa = max(0, x0), xb = min(W, x0 + window);
                const int nx = xb - xa;
                if (!has_player || nx <= 0)
                    continue;
                const int ya = max(0, y0 + r0), yb = min(H, y0 + r1);
                const int ncell = max(0, yb - ya) * nx;
                const CellT *eb = board + ya * W + xa + e * HW;
                uint8_t *ebuf = buf + shift + (size_t)e * patch_bytes +
                                ((size_t)(ya - y0 - r0) * window + (xa - x0)) * C;
                const float inv_nx = 1.0f / (float)nx;
                for (int q = team_tid; q < ncell; q += team) {
                    // q / nx for q < 4096, nx <= 64: (q + 0.5) / nx is at least
                    // 0.5 / nx away from an integer, far beyond float rounding.
                    const int dy = (int)(((float)q + 0.5f) * inv_nx);
                    const int dx = q - dy * nx;
                    uint32_t v = eb[dy * W + dx] & tile_bits;
                    uint8_t *dst = ebuf + ((size_t)dy * window + dx) * C;
                    while (v) {
                        dst[__ffs(v) - 1] = 1;
                        v &= v - 1;
                    }
                }
            }
            if (r0 == 0 && tid < E)
                s_first[pb ^ 1][tid] = HW;  // for the next group (last read two barriers ago)
            fence_async_shared();
            __syncthreads();  // slab complete
            const uint32_t head = min(len, (16u - shift) & 15u);
            const uint32_t mid = (len - head) & ~15u;
            const uint32_t tail = len - head - mid;
            if (tid < head)
                gs[tid] = buf[shift + tid];
            if (tid >= 32 && tid < 32 + tail)
                gs[head + mid + (tid - 32)] = buf[shift + head + mid + (tid - 32)];
            if (tid == 0) {
                if (mid > 0)
                    bulk_store(gs + head, buf + shift + head, mid);
                else
                    asm volatile("cp.async.bulk.commit_group;" ::: "memory");  // keep one group per unit
            }
        }
    }
    if (tid == 0)
        bulk_wait_read<0>();  // shared memory stays valid until the stores have read it
}

// Packed rule record as 32-bit words: [0] h | w << 8, [1] reward,
// [2 + 25p + e] plane p (present, absent, set, clear) at entry e = i*w + k.
constexpr int kRuleWords = 102;

__global__ void rule_obs_kernel(int n_rules_total, int C, const uint32_t *__restrict__ rules,
                                uint8_t *__restrict__ bits, int32_t *__restrict__ reward)
{
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;  // (rule, plane, frame entry)
    if (idx >= n_rules_total * 100)
        return;
    const int rule = idx / 100, p = (idx / 25) & 3, f = idx % 25;
    const uint32_t *rec = rules + (size_t)rule * kRuleWords;
    const int h = (int)(rec[0] & 0xffu), w = (int)((rec[0] >> 8) & 0xffu);
    const int i = f / 5, k = f % 5;
    const uint32_t m = (i < h && k < w) ? rec[2 + 25 * p + i * w + k] : 0u;
    const int NCH = C + 1;
    uint8_t *o = bits + (size_t)idx * NCH;
    for (int c = 0; c < NCH; ++c)
        o[c] = (uint8_t)((m >> c) & 1u);
    if (reward != nullptr && p == 0 && f == 0)
        reward[rule] = (int32_t)rec[1];
}

}  // namespace

int observe_rows_per_slab(int window, int C)
{
    const size_t row_bytes = (size_t)window * C;
    return (int)std::max<size_t>(1, std::min<size_t>((size_t)window, kObsSlabBytes / row_bytes));
}

namespace {

struct ObserveLayout {
    int E, rows, board_region, buf_region;
    size_t smem;
};

// Environments per group: patches up to half of kObsGroupBytes are grouped,
// a power of two of them, up to kObsGroupBytes of patches and
// kObsGroupBoardBytes of boards, keeping at least four groups per SM so that
// every SM has work.
constexpr size_t kObsGroupBytes = 20480;
constexpr size_t kObsGroupBoardBytes = 16384;
// Boards above this size (the band-streamed ones, over 4096 two-byte cells)
// are not staged: the player search and the window's cells read them from
// global memory.
constexpr size_t kObsStageBoardMax = 8192;

ObserveLayout observe_layout(const DevConfig &cf, int window, int sm_count)
{
    ObserveLayout L;
    const size_t patch = (size_t)window * window * cf.C;
    const size_t board = (size_t)cf.HW * cf.cell_bytes;
    size_t E = 1;
    if (patch <= kObsGroupBytes / 2) {
        const size_t cap = std::min<size_t>({(size_t)kObsGroupMax, kObsGroupBytes / patch,
                                             std::max<size_t>(1, kObsGroupBoardBytes / board),
                                             std::max<size_t>(1, (size_t)cf.B / (4 * (size_t)std::max(1, sm_count)))});
        while (2 * E <= cap)  // a power of two, so that teams divide the CTA evenly
            E *= 2;
    }
    L.E = (int)E;
    L.rows = E == 1 ? observe_rows_per_slab(window, cf.C) : window;
    L.board_region = board > kObsStageBoardMax ? 0 : (int)align16(E * board);
    L.buf_region = (int)align16((E == 1 ? (size_t)L.rows * window * cf.C : E * patch) + 16);
    L.smem = 2 * (size_t)L.board_region + 2 * (size_t)L.buf_region;
    return L;
}

int device_sm_count()
{
    static int sm_count = 0;
    if (sm_count == 0) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            sm_count = 1;
    }
    return sm_count;
}

template <typename CellT>
void launch_observe_t(const DevConfig &cf, const CellT *grids, int window, uint8_t *obs, int32_t *player_yx,
                      cudaStream_t st)
{
    const int sm_count = device_sm_count();
    const ObserveLayout L = observe_layout(cf, window, sm_count);
    int per_sm = 1;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, observe_kernel<CellT>, kObsThreads, L.smem) !=
            cudaSuccess ||
        per_sm < 1)
        per_sm = 1;
    const int n_groups = (cf.B + L.E - 1) / L.E;
    const int grid = (int)std::min<long long>(n_groups, (long long)per_sm * sm_count);
    const int vec16 = ((size_t)cf.HW * sizeof(CellT)) % 16 == 0 && (reinterpret_cast<uintptr_t>(grids) & 15u) == 0;
    observe_kernel<CellT><<<grid, kObsThreads, L.smem, st>>>(cf.B, cf.H, cf.W, cf.C, cf.ch_player, grids, window,
                                                             obs, player_yx, L.E, L.rows, L.board_region,
                                                             L.buf_region, vec16);
}

}  // namespace

cudaError_t configure_observe()
{
    cudaError_t e = cudaFuncSetAttribute((const void *)observe_kernel<uint8_t>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute((const void *)observe_kernel<uint16_t>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    return e;
}

void launch_observe(const DevConfig &cf, const void *grids, int window, uint8_t *obs, int32_t *player_yx,
                    cudaStream_t st)
{
    if (cf.cell_bytes == 1)
        launch_observe_t<uint8_t>(cf, (const uint8_t *)grids, window, obs, player_yx, st);
    else
        launch_observe_t<uint16_t>(cf, (const uint16_t *)grids, window, obs, player_yx, st);
}

void launch_rule_obs(int n_rules_total, int C, const uint32_t *rules, uint8_t *bits, int32_t *reward,
                     cudaStream_t st)
{
    const int n = n_rules_total * 100;
    if (n > 0)
        rule_obs_kernel<<<(n + 255) / 256, 256, 0, st>>>(n_rules_total, C, rules, bits, reward);
}

}  // namespace av
