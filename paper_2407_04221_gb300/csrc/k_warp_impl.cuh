// k_warp_impl.cuh -- launchers of the one-warp-per-environment rollout for one
// cell type; included by k_warp_u8.cu and k_warp_u16.cu.
#include "launch.h"

namespace av {
namespace AV_WARP_NS {

template <typename CellT, int NA, int RPW>
void warp_t(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
            const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
            const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
            uint32_t *status, cudaStream_t st)
{
    const int epb = env_warps_per_cta(cf);
    const size_t sm = (size_t)epb * fast_layout(cf).total;
    const int grid = (cf.B + epb - 1) / epb;
    if (cf.rule_words > 0)
        rollout_env_warp_kernel<CellT, NA, RPW, true><<<grid, 32 * epb, sm, st>>>(
            cf, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
            (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
    else
        rollout_env_warp_kernel<CellT, NA, RPW, false><<<grid, 32 * epb, sm, st>>>(
            cf, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
            (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
}

template <typename CellT, int NA>
void warp_na(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
             const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
             const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
             uint32_t *status, cudaStream_t st)
{
#define AV_WARP(RPW)                                                                                    \
    warp_t<CellT, NA, RPW>(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj, \
                           rew_traj, done_traj, rew_sum, status, st)
    if (cf.R <= 2) AV_WARP(2);
    else if (cf.R <= 4) AV_WARP(4);
    else if (cf.R <= 8) AV_WARP(8);
    else AV_WARP(16);
#undef AV_WARP
}

}  // namespace AV_WARP_NS

cudaError_t AV_WARP_CONFIGURE()
{
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    };
#define AV_SETW(CELL, NA, RPW)                                          \
    set((const void *)rollout_env_warp_kernel<CELL, NA, RPW, true>);    \
    set((const void *)rollout_env_warp_kernel<CELL, NA, RPW, false>);
#define AV_SETW_ALL(CELL, NA) AV_SETW(CELL, NA, 2) AV_SETW(CELL, NA, 4) AV_SETW(CELL, NA, 8) AV_SETW(CELL, NA, 16)
    AV_SETW_ALL(AV_WARP_CELL, 1)
    AV_SETW_ALL(AV_WARP_CELL, 2)
#undef AV_SETW_ALL
#undef AV_SETW
    return e;
}

void AV_WARP_LAUNCH(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
                    const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
                    const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj,
                    int32_t *rew_sum, uint32_t *status, cudaStream_t st)
{
    if (cf.NA == 1)
        AV_WARP_NS::warp_na<AV_WARP_CELL, 1>(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                             obs_traj, rew_traj, done_traj, rew_sum, status, st);
    else
        AV_WARP_NS::warp_na<AV_WARP_CELL, 2>(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                             obs_traj, rew_traj, done_traj, rew_sum, status, st);
}

}  // namespace av
