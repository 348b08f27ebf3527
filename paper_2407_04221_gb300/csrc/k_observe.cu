// k_observe.cu -- the policy observation (Sec. 3.2, imitation learning: the
// agent sees a local patch of tiles centred on the player plus a binary form
// of the environment's rules; Sec. 4, Tables 1 and 2: patch widths 5 to 31,
// zero padding outside the map, hidden rules as zeros).
//
// observe_kernel: one CTA per environment.  The board is staged in shared
// memory, the first row-major player cell found by an atomicMin, and the
// patch -- [window][window][C] bytes, channels last -- is built in a shared
// staging slab that is first zero-filled with 16-byte stores; only the set
// bits of the board cells inside the window are then written (a cell holds
// one or two of its C channels, so most bytes are zeros).  The slab's
// 16-byte-aligned middle leaves by one bulk TMA store (cp.async.bulk, shared
// to global); the unaligned head and tail bytes are plain stores, so each
// output byte is written by exactly one CTA whatever the alignment of an
// environment's patch.  Patches larger than the slab go out in row slabs.
//
// rule_obs_kernel: one thread per (rule, plane, frame entry) writes the C + 1
// channel bytes of that entry from the packed 408-byte record.
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

// Wait until the issued bulk stores have read their shared source.
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }

// Wait until the issued bulk stores have completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Make this thread's ordinary shared-memory writes visible to the TMA unit.
__device__ __forceinline__ void fence_async_shared() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

template <typename CellT>
__global__ void __launch_bounds__(kObsThreads)
    observe_kernel(int H, int W, int C, int ch_player, const CellT *__restrict__ grids, int window,
                   uint8_t *__restrict__ obs, int32_t *__restrict__ player_yx, int rows_per_slab)
{
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ int s_first;
    const int HW = H * W;
    CellT *board = reinterpret_cast<CellT *>(smem);
    uint8_t *buf = smem + align16((size_t)HW * sizeof(CellT));
    const int b = blockIdx.x;
    const int tid = threadIdx.x;

    if (tid == 0)
        s_first = HW;
    const CellT *g = grids + (size_t)b * HW;
    for (int q = tid; q < HW; q += kObsThreads)
        board[q] = g[q];
    __syncthreads();
    // The player: the first row-major cell holding the player bit.  A thread
    // scans its cells in increasing order, so its first hit is its minimum.
    for (int q = tid; q < HW; q += kObsThreads)
        if ((board[q] >> ch_player) & 1) {
            atomicMin(&s_first, q);
            break;
        }
    __syncthreads();
    const int first = s_first;
    const bool has_player = first < HW;
    const int py = has_player ? first / W : -1;
    const int px = has_player ? first - (first / W) * W : -1;
    if (player_yx != nullptr && tid == 0) {
        player_yx[2 * b] = py;
        player_yx[2 * b + 1] = px;
    }

    const size_t row_bytes = (size_t)window * C;
    uint8_t *out = obs + (size_t)b * row_bytes * window;
    const int y0 = py - window / 2, x0 = px - window / 2;  // board cell of patch entry (0, 0)
    // Board columns inside the window (the same for every patch row).
    const int xa = max(0, x0), xb = min(W, x0 + window);
    const int nx = xb - xa;
    const uint32_t tile_bits = (1u << C) - 1u;  // bits >= C of a caller's board are not tiles

    for (int r0 = 0; r0 < window; r0 += rows_per_slab) {
        const int r1 = min(window, r0 + rows_per_slab);
        uint8_t *gs = out + (size_t)r0 * row_bytes;
        const uint32_t len = (uint32_t)((size_t)(r1 - r0) * row_bytes);
        const uint32_t shift = (uint32_t)(reinterpret_cast<uintptr_t>(gs) & 15u);  // buf[shift] <-> gs[0]
        const uint32_t words = (shift + len + 15u) >> 4;
        uint4 *buf4 = reinterpret_cast<uint4 *>(buf);
        for (uint32_t j = tid; j < words; j += kObsThreads)
            buf4[j] = make_uint4(0u, 0u, 0u, 0u);
        __syncthreads();
        if (has_player && nx > 0) {
            const int ya = max(0, y0 + r0), yb = min(H, y0 + r1);
            const int ncell = (yb - ya) * nx;
            for (int q = tid; q < ncell; q += kObsThreads) {
                const int dy = q / nx;
                const int y = ya + dy, x = xa + (q - dy * nx);
                uint32_t v = board[y * W + x] & tile_bits;
                uint8_t *dst = buf + shift + ((size_t)(y - y0 - r0) * window + (x - x0)) * C;
                while (v) {
                    dst[__ffs(v) - 1] = 1;
                    v &= v - 1;
                }
            }
        }
        fence_async_shared();
        __syncthreads();
        const uint32_t head = min(len, (16u - shift) & 15u);
        const uint32_t mid = (len - head) & ~15u;
        const uint32_t tail = len - head - mid;
        if (tid < head)
            gs[tid] = buf[shift + tid];
        if (tid >= 32 && tid < 32 + tail)
            gs[head + mid + (tid - 32)] = buf[shift + head + mid + (tid - 32)];
        if (tid == 0 && mid > 0) {
            bulk_store(gs + head, buf + shift + head, mid);
            bulk_wait_read();
        }
        __syncthreads();  // the slab buffer may be rewritten
    }
    if (tid == 0)
        bulk_wait_all();
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

size_t observe_smem_bytes(const DevConfig &cf, int window)
{
    const size_t slab = (size_t)observe_rows_per_slab(window, cf.C) * window * cf.C;
    return align16((size_t)cf.HW * cf.cell_bytes) + align16(slab + 16);
}

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
    const int rows = observe_rows_per_slab(window, cf.C);
    const size_t sm = observe_smem_bytes(cf, window);
    if (cf.cell_bytes == 1)
        observe_kernel<uint8_t><<<cf.B, kObsThreads, sm, st>>>(cf.H, cf.W, cf.C, cf.ch_player,
                                                               (const uint8_t *)grids, window, obs, player_yx, rows);
    else
        observe_kernel<uint16_t><<<cf.B, kObsThreads, sm, st>>>(cf.H, cf.W, cf.C, cf.ch_player,
                                                                (const uint16_t *)grids, window, obs, player_yx,
                                                                rows);
}

void launch_rule_obs(int n_rules_total, int C, const uint32_t *rules, uint8_t *bits, int32_t *reward,
                     cudaStream_t st)
{
    const int n = n_rules_total * 100;
    if (n > 0)
        rule_obs_kernel<<<(n + 255) / 256, 256, 0, st>>>(n_rules_total, C, rules, bits, reward);
}

}  // namespace av
