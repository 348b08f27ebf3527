// k_fast_impl.cuh -- fast rollout launchers for one cell type; included by
// k_fast_u8.cu and k_fast_u16.cu (one translation unit per cell type).
#include "launch.h"

namespace av {
namespace AV_FAST_NS {

template <typename CellT, int NA, int NWARP, int RPW>
void fast_t(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
            const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
            const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
            uint32_t *status, cudaStream_t st)
{
    const size_t sm = fast_layout(cf).total;
    if (cf.rule_words > 0)
        rollout_fast_kernel<CellT, NA, NWARP, RPW, true><<<cf.B, 32 * NWARP, sm, st>>>(
            cf, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
            (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
    else
        rollout_fast_kernel<CellT, NA, NWARP, RPW, false><<<cf.B, 32 * NWARP, sm, st>>>(
            cf, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
            (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
}

// Rules are spread over 4 warps per environment (8 for more than 16 rules, or
// when cf.fast_warps asks for 8).
template <typename CellT, int NA>
void fast_na(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
             const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
             const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
             uint32_t *status, cudaStream_t st)
{
#define AV_FAST(NWARP, RPW)                                                                                \
    fast_t<CellT, NA, NWARP, RPW>(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,    \
                                  obs_traj, rew_traj, done_traj, rew_sum, status, st)
    if (cf.fast_warps == 8 || cf.R > 16) {
        if (cf.R <= 32) AV_FAST(8, 4);
        else AV_FAST(8, 8);
    } else {
        if (cf.R <= 4) AV_FAST(4, 1);
        else if (cf.R <= 8) AV_FAST(4, 2);
        else AV_FAST(4, 4);
    }
#undef AV_FAST
}

}  // namespace AV_FAST_NS

cudaError_t AV_FAST_CONFIGURE()
{
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    };
#define AV_SETF(CELL, NA, NWARP, RPW)                                      \
    set((const void *)rollout_fast_kernel<CELL, NA, NWARP, RPW, true>);    \
    set((const void *)rollout_fast_kernel<CELL, NA, NWARP, RPW, false>);
#define AV_SETF_ALL(CELL, NA) \
    AV_SETF(CELL, NA, 4, 1) AV_SETF(CELL, NA, 4, 2) AV_SETF(CELL, NA, 4, 4) AV_SETF(CELL, NA, 8, 4) AV_SETF(CELL, NA, 8, 8)
    AV_SETF_ALL(AV_FAST_CELL, 1)
    AV_SETF_ALL(AV_FAST_CELL, 2)
#undef AV_SETF_ALL
#undef AV_SETF
    return e;
}

void AV_FAST_LAUNCH(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
                    const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
                    const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj,
                    int32_t *rew_sum, uint32_t *status, cudaStream_t st)
{
    if (cf.NA == 1)
        AV_FAST_NS::fast_na<AV_FAST_CELL, 1>(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                             obs_traj, rew_traj, done_traj, rew_sum, status, st);
    else
        AV_FAST_NS::fast_na<AV_FAST_CELL, 2>(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                             obs_traj, rew_traj, done_traj, rew_sum, status, st);
}

}  // namespace av
