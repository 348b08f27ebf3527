// k_fast_u8.cu -- fast rollout kernels for boards with one byte per cell (C <= 8).
#define AV_FAST_CELL uint8_t
#define AV_FAST_NS fast_u8
#define AV_FAST_CONFIGURE configure_fast_u8
#define AV_FAST_LAUNCH launch_rollout_fast_u8
#include "k_fast_impl.cuh"
