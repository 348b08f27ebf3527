// launch.h -- host-side launchers of libautoverse.so's kernels.  Each group of
// kernels is instantiated in its own translation unit (k_*.cu) so that the
// library builds in parallel.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace av {

// Allow each group's kernels the dynamic shared memory they need.
cudaError_t configure_fast_u8();
cudaError_t configure_fast_u16();
cudaError_t configure_warp_u8();
cudaError_t configure_warp_u16();
cudaError_t configure_block();
cudaError_t configure_expand();
cudaError_t configure_search();
cudaError_t configure_observe();
cudaError_t configure_memo_u8();
cudaError_t configure_memo_u16();
cudaError_t configure_step();

// One step of every environment given its action, one warp per environment
// (k_step.cu): av_step's kernel for boards of at most 16 plane words.
bool use_step_warp(const DevConfig &cf);
void launch_step_warp(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
                      const uint32_t *masks, void *cur, const void *init, int32_t *t, const uint8_t *actions,
                      void *obs, int32_t *rew, uint8_t *done, int32_t *rew_sum, uint32_t *status, cudaStream_t st);

void launch_rollout_fast_u8(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                            const uint32_t *vm, const uint32_t *masks, void *cur, const void *init,
                            int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj,
                            int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                            cudaStream_t st);
void launch_rollout_fast_u16(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                             const uint32_t *vm, const uint32_t *masks, void *cur, const void *init,
                             int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj,
                             int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                             cudaStream_t st);
void launch_rollout_warp_u8(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                            const uint32_t *vm, const uint32_t *masks, void *cur, const void *init,
                            int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj,
                            int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                            cudaStream_t st);
void launch_rollout_warp_u16(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                             const uint32_t *vm, const uint32_t *masks, void *cur, const void *init,
                             int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj,
                             int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                             cudaStream_t st);
void launch_rollout_memo_u8(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                            const uint32_t *vm, const uint32_t *masks, void *cur, const void *init,
                            int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj,
                            int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                            const int32_t *order, uint32_t *cost, cudaStream_t st);
void launch_rollout_memo_u16(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                             const uint32_t *vm, const uint32_t *masks, void *cur, const void *init,
                             int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj,
                             int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                             const int32_t *order, uint32_t *cost, cudaStream_t st);
// Next launch order of the memoising rollout from each environment's cost in
// the last one (k_memo_u16.cu).
void launch_memo_order(const uint32_t *cost, int32_t *order, int B, cudaStream_t st);
void launch_rollout_block(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                          const uint32_t *vm, const uint32_t *masks, void *cur, const void *init, int32_t *t,
                          int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj,
                          int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                          cudaStream_t st);
void launch_expand(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
                   const uint32_t *masks, const void *parents, int F, const int32_t *n_parent, void *children,
                   int32_t *rewards, uint8_t *done, uint64_t *hashes, cudaStream_t st);
void launch_reset(const DevConfig &cf, const uint32_t *cum, uint64_t seed, void *cur, void *init, int32_t *t,
                  void *obs, cudaStream_t st);
void launch_search_init(const DevConfig &cf, uint32_t vmask, const void *roots, uint64_t *root_hash,
                        uint8_t *root_live, uint64_t *vtab, uint32_t *vzero, int32_t *n_visited,
                        cudaStream_t st);
void launch_select_hash(const DevConfig &cf, int cap, uint32_t vmask, int F, const int32_t *n_parent,
                        const int32_t *parent_cum, const uint8_t *parent_live, const void *cand_grids,
                        const int32_t *cand_reward, const uint8_t *cand_done, const uint64_t *cand_hash, int k,
                        void *next_grids, int32_t *next_cum, uint64_t *next_hash, uint8_t *next_live,
                        int32_t *n_next, uint64_t *vtab, uint32_t *vzero, int32_t *n_visited, uint32_t *status,
                        cudaStream_t st);
void launch_select(const DevConfig &cf, int cap, int parity, int F, const int32_t *n_parent,
                   const int32_t *parent_cum, const uint8_t *parent_live, const void *cand_grids,
                   const int32_t *cand_reward, const uint8_t *cand_done, const uint64_t *cand_hash, int k,
                   void *next_grids, int32_t *next_cum, uint64_t *next_hash, uint8_t *next_live,
                   int32_t *n_next, uint64_t *visited, int32_t *n_visited, uint32_t *status, cudaStream_t st);

// Policy observation (k_observe.cu).
int observe_rows_per_slab(int window, int C);
void launch_observe(const DevConfig &cf, const void *grids, int window, uint8_t *obs, int32_t *player_yx,
                    cudaStream_t st);
void launch_rule_obs(int n_rules_total, int C, const uint32_t *rules, uint8_t *bits, int32_t *reward,
                     cudaStream_t st);

// Variant rule semantics (k_variant.cu): apply limits chosen by the largest
// keys of an ordered or random index channel, inhibition masks.
struct VariantParams {
    int32_t random_keys;
    int32_t pad;
    uint64_t key_seed;
    int32_t limit[64];     // 0: every match applies
    uint64_t inhibit[64];  // bit s: a raw match of rule r suppresses rule s
};
cudaError_t configure_variant();
void launch_rollout_variant(const DevConfig &cf, const VariantParams &vp, const uint32_t *arena,
                            const uint32_t *tab_off, const uint32_t *vm, const uint32_t *masks, void *cur,
                            const void *init, int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions,
                            void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum,
                            uint32_t *status, cudaStream_t st);

// Boards larger than one CTA's shared memory (k_band.cu): the step streamed
// through shared memory in bands of rows.
cudaError_t configure_band();
void band_geometry(int H, int W, int *band_rows, int *band_nw, int *na, int *nwp);
void launch_rollout_band(const DevConfig &cf, int band_rows, int band_nw, const uint32_t *arena,
                         const uint32_t *tab_off, const uint32_t *vm, const uint32_t *masks, void *cur,
                         const void *init, int32_t *t, int n_steps, uint64_t seed, const uint8_t *actions,
                         void *obs_traj, int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                         uint32_t *planes, uint32_t *set, uint32_t *clr, uint32_t *base, cudaStream_t st);

// Mutation operators (k_mutate.cu).
void launch_mutate(int B, int H, int W, int C, int R, uint32_t p_map, uint32_t map_channels, uint32_t p_rule,
                   uint32_t p_reward, int32_t reward_min, int32_t reward_max, uint64_t mutable_rules, uint64_t seed,
                   void *maps, uint32_t *rules, cudaStream_t st);

inline cudaError_t configure_kernels()
{
    cudaError_t e = configure_fast_u8();
    if (e == cudaSuccess) e = configure_fast_u16();
    if (e == cudaSuccess) e = configure_warp_u8();
    if (e == cudaSuccess) e = configure_warp_u16();
    if (e == cudaSuccess) e = configure_block();
    if (e == cudaSuccess) e = configure_expand();
    if (e == cudaSuccess) e = configure_search();
    if (e == cudaSuccess) e = configure_observe();
    if (e == cudaSuccess) e = configure_memo_u8();
    if (e == cudaSuccess) e = configure_memo_u16();
    if (e == cudaSuccess) e = configure_step();
    if (e == cudaSuccess) e = configure_variant();
    if (e == cudaSuccess) e = configure_band();
    return e;
}

inline void launch_rollout(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off,
                           const uint32_t *vm, const uint32_t *masks, void *cur, const void *init, int32_t *t,
                           int n_steps, uint64_t seed, const uint8_t *actions, void *obs_traj,
                           int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uint32_t *status,
                           cudaStream_t st, const int32_t *order = nullptr, uint32_t *cost = nullptr)
{
    // A launch of one step given its actions (av_step) has no outcome to
    // repeat: by default it takes the one-warp step kernel (small boards) or
    // the block kernel, whose setups are the shortest.
    if (n_steps == 1 && actions && cf.path == 0) {
        if (use_step_warp(cf))
            launch_step_warp(cf, arena, tab_off, vm, masks, cur, init, t, actions, obs_traj, rew_traj, done_traj,
                             rew_sum, status, st);
        else
            launch_rollout_block(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj,
                                 rew_traj, done_traj, rew_sum, status, st);
        return;
    }
    if (use_memo_rollout(cf) && cf.cell_bytes == 1)
        launch_rollout_memo_u8(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj,
                               rew_traj, done_traj, rew_sum, status, order, cost, st);
    else if (use_memo_rollout(cf))
        launch_rollout_memo_u16(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj,
                                rew_traj, done_traj, rew_sum, status, order, cost, st);
    else if (use_env_warp_rollout(cf) && cf.cell_bytes == 1)
        launch_rollout_warp_u8(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj,
                               rew_traj, done_traj, rew_sum, status, st);
    else if (use_env_warp_rollout(cf))
        launch_rollout_warp_u16(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj,
                                rew_traj, done_traj, rew_sum, status, st);
    else if (use_fast_rollout(cf) && cf.cell_bytes == 1)
        launch_rollout_fast_u8(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj,
                               rew_traj, done_traj, rew_sum, status, st);
    else if (use_fast_rollout(cf))
        launch_rollout_fast_u16(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj,
                                rew_traj, done_traj, rew_sum, status, st);
    else
        launch_rollout_block(cf, arena, tab_off, vm, masks, cur, init, t, n_steps, seed, actions, obs_traj,
                             rew_traj, done_traj, rew_sum, status, st);
}

}  // namespace av
