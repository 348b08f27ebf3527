// k_memo_u16.cu -- memoising rollout for boards with two bytes per cell (C <= 16).
#define AV_MEMO_CELL uint16_t
#define AV_MEMO_NS memo_u16
#define AV_MEMO_CONFIGURE configure_memo_u16
#define AV_MEMO_LAUNCH launch_rollout_memo_u16
#define AV_MEMO_ORDER
#include "k_memo_impl.cuh"
