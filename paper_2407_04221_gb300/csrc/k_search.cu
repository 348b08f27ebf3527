// k_search.cu -- initial maps (reset), search start and best-first selection.
#include "launch.h"

namespace av {

cudaError_t configure_search()
{
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    };
    set((const void *)reset_kernel<uint8_t>);
    set((const void *)reset_kernel<uint16_t>);
    set((const void *)select_kernel<uint8_t>);
    set((const void *)select_kernel<uint16_t>);
    set((const void *)select_hash_kernel<uint8_t>);
    set((const void *)select_hash_kernel<uint16_t>);
    return e;
}

void launch_reset(const DevConfig &cf, const uint32_t *cum, uint64_t seed, void *cur, void *init, int32_t *t,
                  void *obs, cudaStream_t st)
{
    const size_t sm = align16((size_t)cf.HW * 2);
    if (cf.cell_bytes == 1)
        reset_kernel<uint8_t><<<cf.B, kThreads, sm, st>>>(cf, cum, seed, (uint8_t *)cur, (uint8_t *)init, t,
                                                         (uint8_t *)obs);
    else
        reset_kernel<uint16_t><<<cf.B, kThreads, sm, st>>>(cf, cum, seed, (uint16_t *)cur, (uint16_t *)init, t,
                                                          (uint16_t *)obs);
}

void launch_search_init(const DevConfig &cf, uint32_t vmask, const void *roots, uint64_t *root_hash,
                        uint8_t *root_live, uint64_t *vtab, uint32_t *vzero, int32_t *n_visited,
                        cudaStream_t st)
{
    const unsigned grid = (unsigned)((cf.B + kThreads - 1) / kThreads);
    if (cf.cell_bytes == 1)
        search_init_hash_kernel<uint8_t><<<grid, kThreads, 0, st>>>(cf, vmask, (const uint8_t *)roots, root_hash,
                                                                   root_live, vtab, vzero, n_visited);
    else
        search_init_hash_kernel<uint16_t><<<grid, kThreads, 0, st>>>(cf, vmask, (const uint16_t *)roots,
                                                                    root_hash, root_live, vtab, vzero, n_visited);
}

void launch_select_hash(const DevConfig &cf, int cap, uint32_t vmask, int F, const int32_t *n_parent,
                        const int32_t *parent_cum, const uint8_t *parent_live, const void *cand_grids,
                        const int32_t *cand_reward, const uint8_t *cand_done, const uint64_t *cand_hash, int k,
                        void *next_grids, int32_t *next_cum, uint64_t *next_hash, uint8_t *next_live,
                        int32_t *n_next, uint64_t *vtab, uint32_t *vzero, int32_t *n_visited, uint32_t *status,
                        cudaStream_t st)
{
    const size_t sm = select_hash_smem_bytes(F);
    if (cf.cell_bytes == 1)
        select_hash_kernel<uint8_t><<<cf.B, kSelectThreads, sm, st>>>(
            cf, cap, vmask, F, n_parent, parent_cum, parent_live, (const uint8_t *)cand_grids, cand_reward,
            cand_done, cand_hash, k, (uint8_t *)next_grids, next_cum, next_hash, next_live, n_next, vtab, vzero,
            n_visited, status);
    else
        select_hash_kernel<uint16_t><<<cf.B, kSelectThreads, sm, st>>>(
            cf, cap, vmask, F, n_parent, parent_cum, parent_live, (const uint16_t *)cand_grids, cand_reward,
            cand_done, cand_hash, k, (uint16_t *)next_grids, next_cum, next_hash, next_live, n_next, vtab, vzero,
            n_visited, status);
}

void launch_select(const DevConfig &cf, int cap, int parity, int F, const int32_t *n_parent,
                   const int32_t *parent_cum, const uint8_t *parent_live, const void *cand_grids,
                   const int32_t *cand_reward, const uint8_t *cand_done, const uint64_t *cand_hash, int k,
                   void *next_grids, int32_t *next_cum, uint64_t *next_hash, uint8_t *next_live,
                   int32_t *n_next, uint64_t *visited, int32_t *n_visited, uint32_t *status, cudaStream_t st)
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
