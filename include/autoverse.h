/*
 * autoverse.h -- C ABI of libautoverse.so, a batched GPU engine for the
 * rewrite-rule game language of "Autoverse: an Evolvable Game Language for
 * Learning Robust Embodied Agents" (Earle & Togelius, arXiv 2407.04221).
 *
 * Model (Sec. 2.1): a board is an H x W grid of multi-hot cells; bit c of a
 * cell is tile channel c (c < C).  A rewrite rule is an input pattern, an
 * output pattern and a reward (Sec. 2.1, Fig. 2a caption): where the input
 * pattern is present at step t, the output pattern is written at t+1
 * (Sec. 2.1, per-patch definition C_{t+1} = O if the input is present, else
 * C_t), and the rule's reward is paid once per match (Sec. 2.2.1).  All rules
 * apply in parallel to the same board (Sec. 2.1, end of "Possible
 * extensions").  The player acts by placing an invisible force tile next to
 * itself (Sec. 2.1, movement paragraph); force is channel C, visible to rules
 * during the step and never stored.
 *
 * Fixed readings where the paper is silent:
 *  - each rule is matched in 4 rotations (0/90/180/270 degrees CCW: entry
 *    (i,k) of an h x w pattern goes to (w-1-k, i)); every (rule, rotation,
 *    anchor) match counts and pays once;
 *  - only VALID anchors (window fully inside the board);
 *  - conflicting writes: a bit changes when any match asks it to:
 *        next = (F & ~CLR) | (~F & SET), with F the board plus force;
 *  - actions: 0 no-op, 1 up (-y), 2 right (+x), 3 down (+y), 4 left (-x);
 *    values >= 5 act as no-op and raise AV_WARN_ACTION;
 *  - done: no goal tile left (when ch_goal >= 0) or t >= max_steps (when
 *    max_steps > 0); with auto_reset the env returns its own initial map
 *    and t = 0; the observation returned is the board after any reset.
 *
 * Conventions.  Every function returns an int status (AV_OK = 0, negative on
 * error) and never aborts.  Argument checks happen on the host before any
 * launch (AV_EINVAL).  All pointers except av_config, av_rule and init_cum
 * are CALLER-OWNED DEVICE pointers (may be NULL only where stated); work is
 * enqueued on `stream` (a cudaStream_t cast to uintptr_t; 0 = legacy default
 * stream) and returns without synchronising.  Asynchronous CUDA errors are
 * reported by the next call that synchronises (av_sync, av_get_state with a
 * host copy, or any call whose launch fails) as AV_ECUDA; av_last_error()
 * gives the message.  A handle is not thread-safe.  Every call that takes a
 * handle checks that it is alive (returned by av_create and not yet passed to
 * av_destroy): a destroyed or never-created pointer gives AV_ESTATE (a NULL
 * one AV_EINVAL), with no access through it.  av_create returns AV_ENOMEM
 * when a device allocation fails; setting the environment variable
 * AV_FAIL_ALLOC makes every such allocation fail, for testing that path.
 *
 * Board layout in memory ("canonical"): [H][W] cell words, row-major, each
 * cell uint8_t when C <= 8, else uint16_t (little-endian), tile bits only.
 * Batched boards are [B][H][W].
 */
#ifndef AUTOVERSE_H
#define AUTOVERSE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
    AV_OK = 0,
    AV_EINVAL = -1,  /* bad argument, checked before any launch            */
    AV_ENOMEM = -2,  /* device or host allocation failed                   */
    AV_ECUDA = -3,   /* CUDA launch or runtime error                       */
    AV_ESTATE = -4,  /* call not valid in the handle's state, or the handle
                        is not alive (destroyed or never created)          */
    AV_EDEVICE = -5  /* a kernel reported an error through its status word */
};

/* warning bits reported by av_warnings() */
enum { AV_WARN_ACTION = 1 /* an action value >= 5 was treated as no-op */ };

#define AV_MAX_SIDE 256  /* H, W <= 256                                  */
#define AV_MAX_SMEM_CELLS 4096 /* boards of at most this many cells (64 x 64) stay in one
                                  CTA's shared memory and support every call; larger
                                  boards support av_reset, av_set_state, av_get_state,
                                  av_step, av_rollout (streamed in bands of rows,
                                  AV_PATH_BAND), av_observe, av_mutate and av_rule_obs,
                                  and return AV_EINVAL from av_expand, av_search_init,
                                  av_select, av_select_static and av_set_variant with
                                  variants */
#define AV_MAX_C 16      /* C <= 16 tile channels (+1 force channel)     */
#define AV_MAX_PATTERN 5 /* rule patterns up to 5 x 5                    */
#define AV_MAX_RULES 64  /* rules per table                              */
#define AV_MAX_WINDOW 127 /* observation patches up to 127 x 127 (2 * 64 - 1) */

typedef struct av_handle av_handle; /* opaque; owns all env state on the device */

/* Configuration, copied by av_create. */
typedef struct {
    int32_t batch;         /* B >= 1 environments                                   */
    int32_t H, W;          /* 1..AV_MAX_SIDE (see AV_MAX_SMEM_CELLS)                */
    int32_t C;             /* 1..AV_MAX_C tile channels; force is channel C         */
    int32_t n_rules;       /* R rules per table, 0..AV_MAX_RULES                    */
    int32_t rules_per_env; /* 1: rules[B][R]; 0: one table rules[R] for all envs    */
    int32_t max_steps;     /* 0 = no step limit                                     */
    int32_t auto_reset;    /* 1: a done env restores its initial map, t = 0         */
    int32_t ch_player, ch_goal, ch_empty, ch_wall; /* role channels, -1 = none      */
    int32_t border_wall;   /* av_reset: border cells hold only the wall tile        */
    int32_t cum_per_env;   /* 1: init_cum[B][C]; 0: init_cum[C]                     */
    const uint32_t *init_cum; /* HOST pointer, av_reset thresholds: a cell draws u in
                                 [0, 2^24) and takes the first type t with u < cum[t];
                                 copied by av_create; may be NULL (no av_reset)     */
    int32_t search_capacity;  /* av_select: visited hashes kept per env (0 = none)  */
} av_config;

/* Packed rewrite rule, 408 bytes, little-endian (Sec. 2.1: input pattern I,
 * output pattern O, reward).  Entry (i,k) of the h x w base pattern is index
 * i*w + k.  present/absent: bit c (c <= C, bit C = force) must be 1 / 0 at
 * that entry for a match; set/clear: bit c (c < C) written at t+1. */
typedef struct {
    uint8_t h, w;      /* 1..AV_MAX_PATTERN */
    uint8_t _pad[2];
    int32_t reward;    /* paid once per match */
    uint32_t present[25], absent[25], set[25], clear[25];
} av_rule;

/* Create a handle: validates cfg and rules (HOST pointers: rules[B][R] or
 * rules[R] per cfg->rules_per_env), compiles every rule in its 4 rotations
 * and allocates the device state (current boards, initial boards, step
 * counters t, compiled rules).  Boards start all-zero with t = 0 and are
 * their own initial maps until av_reset or av_set_state(set_as_init=1).
 * Returns AV_EINVAL for out-of-range fields, AV_ENOMEM, AV_ECUDA. */
int av_create(const av_config *cfg, const av_rule *rules, av_handle **out);

/* Release the handle and its device memory (after pending work finishes).
 * A NULL handle is AV_EINVAL. */
int av_destroy(av_handle *h);

/* Draw every env's initial map from `seed` (stream 1: cell types from
 * init_cum; stream 2: one player on a uniformly chosen floor cell, or on
 * any interior cell when there is no floor), store it as both the current
 * and the initial map, set t = 0.  obs: device [B][H][W] copy of the maps,
 * or NULL.  AV_ESTATE if the handle has no init_cum. */
int av_reset(av_handle *h, uint64_t seed, void *obs, uintptr_t stream);

/* Replace the current boards (device [B][H][W]); t: device int32[B] or NULL
 * (then t = 0); set_as_init = 1 also makes them the initial maps. */
int av_set_state(av_handle *h, const void *grids, const int32_t *t, int set_as_init,
                 uintptr_t stream);

/* Copy the current boards to device [B][H][W] (and t to device int32[B]
 * when t is not NULL). */
int av_get_state(av_handle *h, void *grids, int32_t *t, uintptr_t stream);

/* One batched step (Sec. 2.1): actions device uint8[B]; obs device
 * [B][H][W] or NULL; reward device int32[B]; done device uint8[B] (reward
 * and done may be NULL).  Updates the handle's boards and t.  An action
 * above 4 acts as 0 and sets AV_WARN_ACTION.  av_step_path names the kernel
 * it launches (one warp per environment for boards of at most 512 cells). */
int av_step(av_handle *h, const uint8_t *actions, void *obs, int32_t *reward, uint8_t *done,
            uintptr_t stream);

/* n_steps fused steps in one launch, boards held on chip.  The action of env
 * b at step s (0-based within this call) is
 *     a = ((draw(action_seed, 4, b, 0, s) >> 32) * 5) >> 32
 * with draw the SplitMix64-keyed counter draw
 *     draw(seed, st, a, b, c) = mix(mix(mix(seed + 0x9E3779B97F4A7C15*(st+1)) ^ a) ^ (b<<32|c)).
 * Optional device outputs (NULL to skip): obs_traj [n_steps][B][H][W],
 * rew_traj int32[n_steps][B], done_traj uint8[n_steps][B], rew_sum int32[B]
 * (sum of this call's rewards). */
int av_rollout(av_handle *h, int32_t n_steps, uint64_t action_seed, void *obs_traj,
               int32_t *rew_traj, uint8_t *done_traj, int32_t *rew_sum, uintptr_t stream);

/* Tree-search expansion (Sec. 2.2.1: the environment is its own forward
 * model for best-first search over player actions): every parent board
 * parents[b][f] (device [B][F][H][W]) stepped by each of the 5 actions with
 * env b's rules -> children [B][F][5][H][W], rewards int32[B][F][5], done
 * uint8[B][F][5] (no goal left; may be NULL) and hashes uint64[B][F][5]
 * (FNV-1a 64 of the child's canonical bytes: offset basis
 * 0xcbf29ce484222325, prime 0x100000001b3).  n_parent: device int32[B] or
 * NULL; when given, parents f >= n_parent[b] are skipped and their output
 * slots are left untouched.  No step counter, no reset: a child is the raw
 * transition.  Stateless with respect to the handle's boards. */
int av_expand(av_handle *h, const void *parents, int32_t F, const int32_t *n_parent,
              void *children, int32_t *rewards, uint8_t *done, uint64_t *hashes,
              uintptr_t stream);

/* Policy observation of each board (Sec. 3.2, imitation learning: the agent
 * observes a local patch of tiles centred on the player's position; Sec. 4,
 * Table 1: patch widths 5, 10, 20 and 31, the map padded with zeros where the
 * patch leaves it).  grids: device [B][H][W] boards, or NULL for the handle's
 * current boards.  obs: device uint8 [B][window][window][C], channels last:
 * byte c of patch entry (i, k) is tile bit c of board cell
 * (py - window/2 + i, px - window/2 + k) (integer division), 0 outside the
 * board; (py, px) is the first row-major cell holding the player bit, and a
 * board without one gives an all-zero patch.  A window of 2 * max(H, W) - 1
 * holds the whole board wherever the player stands.  player_yx: device
 * int32 [B][2] or NULL, receives (py, px), or (-1, -1) without a player.
 * Any alignment of obs is accepted.  AV_EINVAL for window outside
 * 1..AV_MAX_WINDOW or a NULL obs; AV_ESTATE when cfg.ch_player is -1. */
int av_observe(av_handle *h, const void *grids, int32_t window, uint8_t *obs, int32_t *player_yx,
               uintptr_t stream);

/* Binary form of the handle's rule tables (Sec. 3.2: the observation holds a
 * binary representation of the environment's rules; Sec. 4, Table 2 hides
 * them by zeros).  bits: device uint8 [T][R][4][5][5][C+1], T = B when
 * rules_per_env else 1: plane 0 the present and plane 1 the absent entries of
 * the input pattern, plane 2 the set and plane 3 the clear entries of the
 * output pattern; entry (i, k) of the unrotated h x w pattern at frame row i,
 * column k, byte c = channel c (C = force, always 0 in planes 2 and 3), 0
 * outside the pattern.  reward: device int32 [T][R] or NULL, the rules'
 * rewards.  The tables do not change, so one call per handle suffices.
 * AV_EINVAL for a NULL bits with R > 0. */
int av_rule_obs(av_handle *h, uint8_t *bits, int32_t *reward, uintptr_t stream);

#define AV_MAX_LIMIT 255 /* applications per rule per step under av_set_variant */

/* Variant rule semantics (av_set_variant). */
typedef struct {
    int32_t random_keys;             /* 0: ordered index channel; 1: random     */
    int32_t _pad;
    uint64_t key_seed;               /* random index values: counter-draw seed  */
    int32_t limit[AV_MAX_RULES];     /* 0: every match of rule r applies; k: the
                                        k matches with the largest keys          */
    uint64_t inhibit[AV_MAX_RULES];  /* bit s: a raw match of rule r suppresses
                                        rule s for that step                     */
} av_variant;

/* Variant semantics for the handle's av_step and av_rollout (Sec. 2.1,
 * "Possible extensions": a rule may be applied only once or a fixed number of
 * times, and/or in a random order, the tiles to rewrite chosen by the maximum
 * over an additional channel of ordered or random index values; masking lets
 * certain rules inhibit others).  A match is (rule r, rotation j, anchor cell
 * q = y0*W + x0) and has the key (q << 2) | j, or with random_keys
 * ((draw(key_seed, 13, b, t, q) >> 48) << 14) | (q << 2) | j for env b whose
 * step counter is t before the step (draw as for av_rollout's actions), so a
 * rule's matches have distinct keys.  Each step: every rule with at least one
 * match (before limits) suppresses the rules in its inhibit mask; each rule
 * not suppressed applies (writes, pays) its limit[r] matches with the largest
 * keys, or all of them when limit[r] is 0; the writes then combine as in the
 * standard step.  v = NULL, or all limits and masks zero, restores the standard
 * step.  While variants are set, av_rollout_path reports AV_PATH_VARIANT and
 * av_expand returns AV_ESTATE.  AV_EINVAL for a limit outside 0..AV_MAX_LIMIT,
 * random_keys not 0 or 1, or a limit or mask bit naming a rule slot >= n_rules.
 * Host call; takes effect for work enqueued after it. */
int av_set_variant(av_handle *h, const av_variant *v);

/* Rates and ranges of the mutation operators (av_mutate). */
typedef struct {
    uint32_t p_map;         /* map bit flip rate x 2^24 (0..2^24)                       */
    uint32_t map_channels;  /* bit c: tile channel c of the maps may flip               */
    uint32_t p_rule;        /* rule entry change rate x 2^24 (0..2^24)                  */
    uint32_t p_reward;      /* reward redraw rate x 2^24 (0..2^24)                      */
    int32_t reward_min, reward_max; /* redrawn rewards are uniform in [min, max]        */
    uint64_t mutable_rules; /* bit r: rule slot r of every table may mutate             */
} av_mutation;

/* Mutation operators of the evolution loop (Sec. 3.1.1: the initial map, a
 * multi-hot array, is mutated by flipping bits; the mutable rules by changing
 * tiles of their input and/or output patterns at any position; rewards may
 * change too, to positive or negative values).  In place, on caller-owned
 * device arrays, without a handle:
 *   maps:  device [batch][H][W] cell words (uint8 when C <= 8, else uint16),
 *          or NULL: bit c of cell q = y*W + x of env b flips when
 *          draw(seed, 9, b, q, c) >> 40 < p_map and bit c of map_channels is set;
 *   rules: device av_rule [batch][n_rules], or NULL: for every rule slot r in
 *          mutable_rules, every entry e < h*w of the input pattern (channels
 *          0..C, force included; states don't-care / present / absent) and
 *          of the output pattern (channels 0..C-1; states unchanged / set /
 *          clear) changes when d >> 40 < p_rule, d = draw(seed, 10 (input) or
 *          11 (output), b, 25 r + e, c), to the next state cyclically when
 *          bit 39 of d is 0, else to the one after; the reward becomes
 *          reward_min + ((draw(seed, 12, b, r, 1) >> 32) * n >> 32),
 *          n = reward_max - reward_min + 1, when draw(seed, 12, b, r, 0) >> 40
 *          < p_reward.  Pattern sizes do not change.
 * draw is the counter draw of av_rollout.  Records must be valid (as av_create
 * checks); mutated records stay valid.  A new handle made from the mutated
 * records (av_create, host copies) and maps (av_set_state with set_as_init)
 * evaluates the offspring.  AV_EINVAL for sizes outside the av_config limits,
 * a NULL m, a rate above 2^24 or reward_min > reward_max. */
int av_mutate(int32_t batch, int32_t H, int32_t W, int32_t C, int32_t n_rules, const av_mutation *m,
              uint64_t seed, void *maps, av_rule *rules, uintptr_t stream);

/* Start a search from the root boards roots (device [B][H][W]): writes
 * root_hash uint64[B] (FNV-1a 64 as in av_expand) and root_live uint8[B]
 * (1 unless the root has no goal left), and sets the visited set of env b
 * to { root_hash[b] }.  AV_ESTATE if cfg.search_capacity < 1.  The handle
 * keeps each env's visited set as an open-addressing hash table of the
 * smallest power of two >= max(64, 2 x search_capacity) 8-byte slots. */
int av_search_init(av_handle *h, const void *roots, uint64_t *root_hash, uint8_t *root_live,
                   uintptr_t stream);

/* One selection step of greedy best-first search (Sec. 2.2.1: states equal
 * to an earlier one are pruned, keeping the shallower; of equal states the
 * higher reward is kept).  Candidates are the children of av_expand for F
 * parents per env: cand_grids [B][F][5][H][W], cand_reward int32[B][F][5],
 * cand_done uint8[B][F][5], cand_hash uint64[B][F][5]; parent_cum int32[B][F]
 * and parent_live uint8[B][F] (a candidate exists only for parent f <
 * n_parent[b] with parent_live != 0; n_parent int32[B]).  Per env:
 * cum = parent_cum + reward; drop hashes already visited; among equal
 * hashes keep the highest cum (then the lowest candidate index); rank by
 * (cum desc, hash asc); keep the first min(k, count) as the next frontier
 * next_grids [B][k][H][W], next_cum int32[B][k], next_hash uint64[B][k],
 * next_live uint8[B][k] (= !done), n_next int32[B]; add their hashes to the
 * visited set.  AV_EINVAL if 5*F > 4096 or k > 5*F; AV_EDEVICE (via
 * av_sync) if a visited set would exceed search_capacity. */
int av_select(av_handle *h, int32_t F, const int32_t *n_parent, const int32_t *parent_cum,
              const uint8_t *parent_live, const void *cand_grids, const int32_t *cand_reward,
              const uint8_t *cand_done, const uint64_t *cand_hash, int32_t k, void *next_grids,
              int32_t *next_cum, uint64_t *next_hash, uint8_t *next_live, int32_t *n_next,
              uintptr_t stream);

/* Largest 2 * batch * capacity accepted by av_select_static (hashes). */
#define AV_SELECT_STATIC_MAX_HASHES (1 << 21) /* 16 MiB of uint64 */

/* av_select without a handle and without allocating anything.  For callers
 * that cannot call cudaMalloc: code running under an allocator they do not
 * own, inside a memory pool with a fixed budget, or in a process where a
 * device allocation would break their own memory accounting.  The paper has
 * no counterpart: this is a deployment variant of av_select.
 *
 * Same selection as av_select for boards of batch x H x W cells with C tile
 * channels; the visited sets are caller-owned: visited uint64[batch][capacity]
 * (device, env b's first n_visited[b] entries sorted ascending) and n_visited
 * int32[batch] (device), both updated in place; entries past an env's new
 * count are left as they were.  status: device uint32 or NULL; it is
 * overwritten with this call's bits: bit 0 when a visited set would exceed
 * capacity (that env's set and count are left unchanged), bit 1 when an
 * n_visited[b] lies outside 0..capacity (that env selects nothing: n_next[b]
 * = 0, its frontier zeroed, its set and count left unchanged).
 *
 * The working copy of the visited sets lives in one file-scope device array
 * of AV_SELECT_STATIC_MAX_HASHES hashes that every GPU loading the library
 * holds until the process exits; sizes with 2 * batch * capacity above it
 * are rejected with AV_EINVAL before any GPU work.  The first call on a
 * device looks up the array's device address (with that device current):
 * make that first call before any stream capture.  All calls share the
 * array, so calls that overlap on the GPU (other streams, other threads)
 * race: serialise them.  No cudaMalloc, cudaFree or other allocation is
 * made; the work is enqueued on `stream`. */
int av_select_static(int32_t batch, int32_t H, int32_t W, int32_t C, int32_t F,
                     const int32_t *n_parent, const int32_t *parent_cum,
                     const uint8_t *parent_live, const void *cand_grids,
                     const int32_t *cand_reward, const uint8_t *cand_done,
                     const uint64_t *cand_hash, int32_t k, void *next_grids, int32_t *next_cum,
                     uint64_t *next_hash, uint8_t *next_live, int32_t *n_next, uint64_t *visited,
                     int32_t *n_visited, int32_t capacity, uint32_t *status, uintptr_t stream);

/* Wait for the handle's pending work (device-wide synchronise) and report
 * deferred errors: AV_ECUDA for a CUDA error, AV_EDEVICE when a kernel set
 * its error status (e.g. visited set overflow). */
int av_sync(av_handle *h);

/* Warning bits seen since the last call (synchronises); see AV_WARN_*. */
int av_warnings(av_handle *h, uint32_t *bits);

/* Which rollout kernel av_step / av_rollout launch for this handle:
 * AV_PATH_MEMO (boards of at most 512 cells, any rule count: one CTA per
 * environment that evaluates each (board, action) pair once and repeats its
 * outcome while the board stays unchanged), AV_PATH_BLOCK (one CTA per
 * environment, every step evaluated; larger boards), AV_PATH_VARIANT when
 * variant semantics are set (av_set_variant), or AV_PATH_BAND for boards of
 * more than AV_MAX_SMEM_CELLS cells (one CTA per environment streams the
 * board through shared memory in bands of rows).  AV_PATH_FAST (several warps
 * per environment, boards of at most 512 cells and at most 64 rules) and
 * AV_PATH_WARP (one warp per environment, boards of at most 512 cells and at
 * most 16 rules) step every environment every step; they run when the
 * environment variable AV_KERNEL_PATH=block|fast|warp|memo, read by av_create,
 * forces a path for tests and measurements.  Every path gives the same
 * results.  The path named is av_rollout's; av_step's is av_step_path's.
 * Writes the path to *path; AV_EINVAL for a null argument.  No GPU work. */
enum { AV_PATH_BLOCK = 1, AV_PATH_FAST = 2, AV_PATH_WARP = 3, AV_PATH_VARIANT = 4, AV_PATH_BAND = 5,
       AV_PATH_MEMO = 6, AV_PATH_STEP = 7 };
int av_rollout_path(av_handle *h, int32_t *path);

/* Which kernel av_step launches for this handle (Sec. 2.1, one step of every
 * environment given its action): AV_PATH_STEP (one warp per environment,
 * eight environments per CTA, the rule table read where it lies: boards of at
 * most 512 cells), AV_PATH_BLOCK (larger boards, up to 64 x 64), or, with
 * variant semantics set, boards in bands, or AV_KERNEL_PATH forcing a path,
 * the kernel av_rollout_path names.  Every path gives the same results.
 * Writes the path to *path; AV_EINVAL for a null argument.  No GPU work. */
int av_step_path(av_handle *h, int32_t *path);

/* Static description of a status code. */
const char *av_strerror(int status);

/* Message of the handle's last error ("" if none); valid until the next call. */
const char *av_last_error(av_handle *h);

#ifdef __cplusplus
}
#endif

#endif /* AUTOVERSE_H */
