// k_fast_u16.cu -- fast rollout kernels for boards with two bytes per cell (C > 8).
#define AV_FAST_CELL uint16_t
#define AV_FAST_NS fast_u16
#define AV_FAST_CONFIGURE configure_fast_u16
#define AV_FAST_LAUNCH launch_rollout_fast_u16
#include "k_fast_impl.cuh"
