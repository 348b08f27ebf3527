// k_warp_u16.cu -- one-warp-per-environment rollout for boards with two bytes per cell (C <= 16).
#define AV_WARP_CELL uint16_t
#define AV_WARP_NS warp_u16
#define AV_WARP_CONFIGURE configure_warp_u16
#define AV_WARP_LAUNCH launch_rollout_warp_u16
#include "k_warp_impl.cuh"
