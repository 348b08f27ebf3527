// k_memo_u8.cu -- memoising rollout for boards with one byte per cell (C <= 8).
#define AV_MEMO_CELL uint8_t
#define AV_MEMO_NS memo_u8
#define AV_MEMO_CONFIGURE configure_memo_u8
#define AV_MEMO_LAUNCH launch_rollout_memo_u8
#include "k_memo_impl.cuh"
