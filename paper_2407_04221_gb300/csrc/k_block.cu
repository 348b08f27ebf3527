// k_block.cu -- rollout kernels with one CTA of kThreads per environment, any
// board size (used for boards of more than 16 plane words).
#include "launch.h"

namespace av {
namespace {

#define AV_FOR_NA(MACRO, CELL) MACRO(CELL, 1) MACRO(CELL, 2) MACRO(CELL, 4) MACRO(CELL, 8) MACRO(CELL, 16)

template <typename CellT, int NA, bool SM>
void block_launch(const DevConfig &cf, size_t sm, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
                  const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
                  const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
                  uint32_t *status, cudaStream_t st)
{
    // one-step launches of small boards (av_step) take the kernel without runs
    if constexpr (NA <= 2) {
        if (n_steps == 1) {
            rollout_kernel<CellT, NA, SM, false><<<cf.B, kThreads, sm, st>>>(
                cf, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
                (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
            return;
        }
    }
    rollout_kernel<CellT, NA, SM, true><<<cf.B, kThreads, sm, st>>>(
        cf, arena, tab_off, vm, masks, (CellT *)cur, (const CellT *)init, t, n_steps, seed, actions,
        (CellT *)obs_traj, rew_traj, done_traj, rew_sum, status);
}

template <typename CellT, int NA>
void block_t(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
             const uint32_t *masks, void *cur, const void *init, int32_t *t, int n_steps, uint64_t seed,
             const uint8_t *actions, void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
             uint32_t *status, cudaStream_t st)
{
    const size_t sm = step_smem(cf, 0).total;
    if (cf.rule_words > 0)
        block_launch<CellT, NA, true>(cf, sm, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                      obs_traj, rew_traj, done_traj, rew_sum, status, st);
    else
        block_launch<CellT, NA, false>(cf, sm, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions,
                                       obs_traj, rew_traj, done_traj, rew_sum, status, st);
}

}  // namespace

cudaError_t configure_block()
{
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    };
#define AV_SET(CELL, NA)                                       \
    set((const void *)rollout_kernel<CELL, NA, true, true>);   \
    set((const void *)rollout_kernel<CELL, NA, false, true>);  \
    if (NA <= 2) {                                             \
        set((const void *)rollout_kernel<CELL, NA, true, NA <= 2 ? false : true>);  \
        set((const void *)rollout_kernel<CELL, NA, false, NA <= 2 ? false : true>); \
    }
    AV_FOR_NA(AV_SET, uint8_t)
    AV_FOR_NA(AV_SET, uint16_t)
#undef AV_SET
    return e;
}

void launch_rollout_block(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                          const uint32_t *vm, const uint32_t *masks, void *cur, const void *init, int32_t *t,
                          int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj,
                          int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                          cudaStream_t st)
{
#define AV_CASE(CELL, NA)                                                                              \
    case NA:                                                                                          \
        block_t<CELL, NA>(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj, \
                          rew_traj, done_traj, rew_sum, status, st);                                  \
        break;
    if (cf.cell_bytes == 1) {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint8_t) }
    } else {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint16_t) }
    }
#undef AV_CASE
}

}  // namespace av
