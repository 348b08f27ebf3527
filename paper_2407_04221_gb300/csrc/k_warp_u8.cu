// k_warp_u8.cu -- one-warp-per-environment rollout for boards with one byte per cell (C <= 8).
#define AV_WARP_CELL uint8_t
#define AV_WARP_NS warp_u8
#define AV_WARP_CONFIGURE configure_warp_u8
#define AV_WARP_LAUNCH launch_rollout_warp_u8
#include "k_warp_impl.cuh"
