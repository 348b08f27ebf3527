// k_expand.cu -- tree-search expansion kernels: one warp per parent for boards
// of at most 16 plane words, one CTA per parent otherwise.
#include "launch.h"

namespace av {
namespace {

#define AV_FOR_NA(MACRO, CELL) MACRO(CELL, 1) MACRO(CELL, 2) MACRO(CELL, 4) MACRO(CELL, 8) MACRO(CELL, 16)

// Parents per CTA on the warp path: 1 while the GPU has room for every warp at
// once (best balance), more for large batches.  The count divides F so that
// a CTA's parents share one environment (and its rule table).
int warps_per_cta(long long units, int F)
{
    int w = units <= 152LL * 32 ? 1 : (units <= 152LL * 64 ? 2 : kWarpCtaMax);
    while (w > 1 && F % w != 0)
        w >>= 1;
    return w;
}

template <typename CellT, int NA>
void block_t(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
             const uint32_t *masks, const void *parents, int F, const int32_t *n_parent, void *children,
             int32_t *rewards, uint8_t *done, uint64_t *hashes, cudaStream_t st)
{
    const size_t sm = step_smem(cf, 5).total;
    const unsigned grid = (unsigned)(cf.B * F);
    if (cf.rule_words > 0)
        expand_kernel<CellT, NA, true><<<grid, kThreads, sm, st>>>(cf, arena, tab_off, vm, masks,
                                                                  (const CellT *)parents, F, n_parent,
                                                                  (CellT *)children, rewards, done, hashes);
    else
        expand_kernel<CellT, NA, false><<<grid, kThreads, sm, st>>>(cf, arena, tab_off, vm, masks,
                                                                   (const CellT *)parents, F, n_parent,
                                                                   (CellT *)children, rewards, done, hashes);
}

template <typename CellT, int NA>
void warp_t(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
            const uint32_t *masks, const void *parents, int F, const int32_t *n_parent, void *children,
            int32_t *rewards, uint8_t *done, uint64_t *hashes, cudaStream_t st)
{
    const long long units = (long long)cf.B * F;
    const int wpc = warps_per_cta(units, F);
    const unsigned grid = (unsigned)((units + wpc - 1) / wpc);
    const ExpandLayout L = expand_layout(cf);
    const size_t sm = L.warps + (size_t)wpc * L.per_warp;
    if (cf.rule_words > 0)
        expand_warp_kernel<CellT, NA, true><<<grid, 32 * wpc, sm, st>>>(
            cf, arena, tab_off, vm, masks, (const CellT *)parents, F, n_parent, (CellT *)children, rewards,
            done, hashes);
    else
        expand_warp_kernel<CellT, NA, false><<<grid, 32 * wpc, sm, st>>>(
            cf, arena, tab_off, vm, masks, (const CellT *)parents, F, n_parent, (CellT *)children, rewards,
            done, hashes);
}

}  // namespace

cudaError_t configure_expand()
{
    cudaError_t e = cudaSuccess;
    auto set = [&](const void *fn) {
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmemLimit);
    };
#define AV_SET(CELL, NA)                                      \
    set((const void *)expand_kernel<CELL, NA, true>);         \
    set((const void *)expand_kernel<CELL, NA, false>);
    AV_FOR_NA(AV_SET, uint8_t)
    AV_FOR_NA(AV_SET, uint16_t)
#undef AV_SET
#define AV_SETW(CELL, NA)                                            \
    set((const void *)expand_warp_kernel<CELL, NA, true>);           \
    set((const void *)expand_warp_kernel<CELL, NA, false>);
    AV_SETW(uint8_t, 1)
    AV_SETW(uint8_t, 2)
    AV_SETW(uint16_t, 1)
    AV_SETW(uint16_t, 2)
#undef AV_SETW
    return e;
}

void launch_expand(const DevConfig &cf, const uint32_t *arena, const uint32_t *tab_off, const uint32_t *vm,
                   const uint32_t *masks, const void *parents, int F, const int32_t *n_parent, void *children,
                   int32_t *rewards, uint8_t *done, uint64_t *hashes, cudaStream_t st)
{
    const bool u8 = cf.cell_bytes == 1;
    if (use_warp_expand(cf)) {
        if (cf.NA == 1) {
            if (u8)
                warp_t<uint8_t, 1>(cf, arena, tab_off, vm, masks, parents, F, n_parent, children, rewards, done,
                                      hashes, st);
            else
                warp_t<uint16_t, 1>(cf, arena, tab_off, vm, masks, parents, F, n_parent, children, rewards,
                                       done, hashes, st);
        } else {
            if (u8)
                warp_t<uint8_t, 2>(cf, arena, tab_off, vm, masks, parents, F, n_parent, children, rewards, done,
                                      hashes, st);
            else
                warp_t<uint16_t, 2>(cf, arena, tab_off, vm, masks, parents, F, n_parent, children, rewards,
                                       done, hashes, st);
        }
        return;
    }
#define AV_CASE(CELL, NA)                                                                               \
    case NA:                                                                                           \
        block_t<CELL, NA>(cf, arena, tab_off, vm, masks, parents, F, n_parent, children, rewards, done, \
                          hashes, st);                                                                 \
        break;
    if (u8) {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint8_t) }
    } else {
        switch (cf.NA) { AV_FOR_NA(AV_CASE, uint16_t) }
    }
#undef AV_CASE
}

}  // namespace av
