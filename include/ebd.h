/*
 * ebd.h -- C ABI of the Early-Bird (EB) decoding step on one GB300 GPU.
 *
 * One call of ebd_step() performs one denoising step of EB decoding over
 * the active window of every sequence in a batch (paper arxiv 2609.16450):
 *
 *   1. window attention: the window's queries attend bidirectionally to the
 *      cached prefix keys/values followed by the window's own keys/values
 *      (Sec. 3 "bidirectional Transformer"; Sec. 6.3 "Effect of KV-Cache
 *      Configuration", prefix cache at the block boundary);
 *   2. the LM head l = W_lm h for every window row, reduced on the fly to
 *      the per-position statistics of the softmax (App. B Eq. app-confidence:
 *      kappa = max_v p(v); Sec. 5.1: normalized entropy H~ and top-1 token
 *      x_hat; Sec. 5.2: top-1/top-2 gap Delta); logits never reach memory;
 *   3. the EB decision (App. E, algorithm "Inference with LBS Block
 *      Selection and LPS Parallel Commit"): when a sequence has no active
 *      block, the LBS router (Sec. 5.1, App. C.1 Eq. lbs_feat) scores its
 *      masked rows and the filters (EOS removal, max gap g_max, min tokens
 *      L_min with the first-L_B fallback) select the block; the LPS router
 *      (Sec. 5.2, App. D.1) scores the block's masked rows; the union accept
 *      rule (kappa >= tau or p_psi > tau_psi), the anti-stall fallback and the
 *      parallel commit update tokens, mask and block state in place.
 *
 * Conventions
 *   - bf16 tensors are passed as uint16_t bit patterns, row-major, densely
 *     packed, 16-byte aligned.  Every pointer in ebd_step_args is a DEVICE
 *     pointer on the handle's device, owned by the caller, except in
 *     ebd_step_host() (see there).
 *   - The handle owns the router weights, the folded token-branch table,
 *     a workspace and a device status word; nothing else is allocated per
 *     call.  One handle serves one stream at a time; it is not thread-safe.
 *   - Functions that take a stream only enqueue work (asynchronous); they
 *     check their arguments on the host first and return an error without
 *     enqueuing anything when a check fails.  Failures detected on the
 *     device (a bounded wait that gave up, a non-finite logit statistic, an
 *     inconsistent row count) are recorded in the status word and reported
 *     by ebd_sync_status().
 *   - Supported shapes: d_model % 8 == 0, d_base % 8 == 0, head_dim in
 *     {64, 128}, n_heads_q % n_heads_kv == 0, 1 <= window rows of a
 *     sequence <= max_window <= 512, gen_len >= max_window, vocab >= 2,
 *     rows of a step <= max_rows <= 4096.  Anything else returns
 *     EBD_ERR_UNSUPPORTED.
 *   - max_window <= 64: the decision runs as one thread-block cluster per
 *     sequence; with max_window <= 32, a launch of 16 or more sequences runs
 *     it as one CTA per sequence instead (the same results; the environment
 *     variable EBD_DECIDE_KERNEL = "cta" or "cluster" forces either kernel
 *     for max_window <= 32).  max_window > 64 (the full-sequence setting, where every
 *     position of the response is a row, App. E with M = all masked
 *     positions): the decision runs as a chain of grid-wide kernels, and a
 *     step takes no window attention (attn_out and kv_append must be unset:
 *     EBD_ERR_UNSUPPORTED otherwise).
 *   - stream arguments are cudaStream_t values passed as void* (NULL = the
 *     legacy default stream).
 */
#ifndef EBD_H_
#define EBD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct ebd_handle ebd_handle;

typedef int32_t ebd_status;
#define EBD_OK 0
#define EBD_ERR_INVALID_ARG (-1) /* null pointer, bad size, misalignment    */
#define EBD_ERR_UNSUPPORTED (-2) /* shape outside the supported set          */
#define EBD_ERR_CUDA (-3)        /* a CUDA runtime/driver call failed        */
#define EBD_ERR_TIMEOUT (-4)     /* a device-side bounded wait gave up       */
#define EBD_ERR_NONFINITE (-5)   /* NaN/Inf logit statistic; row not committed */
#define EBD_ERR_STATE (-6)       /* call order: e.g. LBS needs a bound W_e   */
#define EBD_ERR_BOUNDS (-7)      /* checked builds (EBD_CHECKS) only: a device
                                    index outside its buffer; the access was
                                    skipped                                   */

/* decode_mode: which decision step 3 applies.  EBD_DECODE_EB is the EB
 * decision (LBS + LPS, App. E).  The other two are the fixed-block update
 * of the baselines (App. B, Eq. prelim-update) on the rows of the window,
 * which the caller sets to the active fixed block (see
 * ebd_loop_block_window); the routers do not run and the block state is
 * left untouched.  THRESHOLD commits the masked rows with kappa >= tau, or
 * the one with the highest kappa when none reaches tau (Fast-dLLM's rule).
 * TOPM commits the min(top_m, |M|) masked rows with the highest kappa (the
 * vanilla budget rule); ties go to the lower position in both. */
#define EBD_DECODE_EB 0
#define EBD_DECODE_THRESHOLD 1
#define EBD_DECODE_TOPM 2

/* debug_flags bits (tests only) */
#define EBD_DEBUG_FORCE_TIMEOUT 1 /* LM-head kernel waits on a barrier that
                                     nothing completes, with a 20 ms limit */
#define EBD_DEBUG_FORCE_COPY_TIMEOUT 2 /* ebd_step_host: the attention waits for
                                     a copy-stream ticket that is never
                                     written, with a 20 ms limit */

typedef struct {
  /* backbone shapes */
  int32_t d_model;     /* hidden size d                                     */
  int32_t vocab;       /* |V|                                               */
  int32_t n_heads_q;   /* query heads Hq                                    */
  int32_t n_heads_kv;  /* key/value heads Hkv (GQA when < Hq)               */
  int32_t head_dim;    /* D                                                 */
  int32_t d_base;      /* width of the frozen token embedding W_e           */
  /* capacity of the handle */
  int32_t max_batch;   /* sequences per step                                */
  int32_t max_window;  /* window rows per sequence (<= 512; > 64: the
                          full-sequence setting, see above)                 */
  int32_t max_rows;    /* window rows per step, all sequences (<= 4096)     */
  int32_t max_prefix;  /* P_max: second dimension of the K/V cache          */
  /* EB hyper-parameters (App. F) */
  int32_t gen_len;     /* L: rows of the LBS positional table E_pos         */
  int32_t g_max;       /* max gap between consecutive block members (5)     */
  int32_t l_min;       /* min block size (8 LLaDA/Dream, 16 LLaDA-1.5)      */
  int32_t l_b;         /* min-tokens fallback block size (32)               */
  int32_t eos_id;      /* token id removed from LBS candidates              */
  int32_t lps_enabled; /* 1: union accept with LPS; 0: LBS + threshold only */
  float tau;           /* confidence threshold (0.9)                        */
  float tau_psi;       /* LPS acceptance threshold (0.89 / 0.90 / 0.87)     */
  uint64_t seed;       /* seed of the routers' random init                  */
  int32_t debug_flags; /* EBD_DEBUG_* (tests); 0 in normal use              */
  int32_t decode_mode; /* EBD_DECODE_*: EB decision or a baseline rule      */
  int32_t top_m;       /* EBD_DECODE_TOPM: commits per step (>= 1)          */
  int32_t reserved;
} ebd_config;

typedef struct {
  int32_t batch;              /* B <= max_batch                                  */
  int32_t rows;               /* R = cu_rows[B] <= max_rows (host copy)          */
  const int32_t* cu_rows;     /* [B+1] window row offsets, cu_rows[0] = 0        */
  const int32_t* prefix_len;  /* [B] cached prefix length, <= max_prefix         */
  const int32_t* row_pos;     /* [R] absolute position of each window row,
                                 strictly increasing within a sequence         */
  const uint16_t* hidden;     /* [R][d_model] bf16 final hidden states           */
  const uint16_t* q;          /* [R][Hq][D] bf16 window queries                  */
  const uint16_t* k_win;      /* [R][Hkv][D] bf16 window keys                    */
  const uint16_t* v_win;      /* [R][Hkv][D] bf16 window values                  */
  uint16_t* k_cache;          /* [B][max_prefix][Hkv][D] bf16 K/V cache, indexed by
                                 absolute position: the prefix [0, prefix_len),
                                 the suffix range (dual cache); written only
                                 when kv_append is set                         */
  uint16_t* v_cache;          /* [B][max_prefix][Hkv][D] bf16 cached values      */
  const uint16_t* w_lm;       /* [vocab][d_model] bf16 LM-head weight            */
  /* decode state, read and updated in place */
  int32_t* tokens;            /* [R] token ids; committed rows get x_hat         */
  uint8_t* mask;              /* [R] 1 = [MASK]; committed rows become 0         */
  uint8_t* in_block;          /* [R] 1 = member of the active block B            */
  int32_t* blk_meta;          /* [B][2] {b = min position of B, |B| at selection};
                                 |B| = 0 means no active block                 */
  /* outputs; any of them may be NULL */
  float* attn_out;            /* [R][Hq][D] fp32 attention output                */
  float* conf;                /* [R] kappa                                       */
  float* entropy;             /* [R] H in nats                                   */
  float* ent_norm;            /* [R] H~ = H / ln(vocab)                          */
  float* gap;                 /* [R] Delta = p(top1) - p(top2)                   */
  int32_t* argmax;            /* [R] x_hat (lowest index on ties)                */
  float* lbs_logit;           /* [R] O_phi where LBS ran, NaN elsewhere          */
  float* lps_prob;            /* [R] p_psi where LPS scored, NaN elsewhere       */
  uint8_t* accepted;          /* [R] 1 = committed this step                     */
  int32_t w_lm_layout;        /* 0: w_lm is [vocab][d_model] row-major;
                                 1: w_lm is the tiled copy written by
                                 ebd_pack_lm_head()                           */
  /* KV-cache integration (Sec. 6.3, prefix and dual cache) */
  int32_t kv_append;          /* 1: after the decision, every window row that is
                                 committed (mask 0 after the step) has its
                                 k_win/v_win row written into k_cache/v_cache
                                 at row_pos (the prefix-cache append on
                                 commit); rows at positions >= max_prefix are
                                 skipped.  It runs after the step's window
                                 attention, which reads the cache as it was
                                 before.  0: the cache is only read.          */
  const int32_t* suffix;      /* [B][2] {s0, S}, device (host in
                                 ebd_step_host): the window also attends to
                                 the cached keys/values at positions
                                 [s0, s0 + S) after its own (dual cache).  The
                                 range is clamped to [0, max_prefix) and must
                                 not overlap the window's positions.  NULL:
                                 prefix cache only.                           */
} ebd_step_args;

/* Creates a handle on the current CUDA device: validates *cfg, allocates the
 * router weights (random-init from cfg->seed, see ebd_router_init_host),
 * the workspace and the status word.  On failure *out is NULL. */
ebd_status ebd_create(const ebd_config* cfg, ebd_handle** out);

/* Frees everything the handle owns (never caller memory).  NULL-safe.
 * Synchronises the device first. */
void ebd_destroy(ebd_handle* h);

/* Binds the frozen token embedding W_e [vocab][d_base] bf16 (device,
 * caller-owned; it must stay valid while bound) and folds the LBS token
 * branch: table[v] = W_tok W_e[v] (App. C.1 "Token branch"; the projection
 * is linear, so it is applied to every vocabulary row once instead of to the
 * gathered rows of every step).  Must precede any step in which LBS runs;
 * ebd_import_weights() re-folds with the bound table.  Enqueued on stream. */
ebd_status ebd_bind_embedding(ebd_handle* h, const uint16_t* w_emb, void* stream);

/* Size in bytes of the tiled LM-head weight written by ebd_pack_lm_head():
 * ceil(vocab/64) * ceil(d_model/64) tiles of 64 x 64 bf16. */
size_t ebd_lm_head_packed_bytes(const ebd_config* cfg);

/* Writes W_lm ([vocab][d_model] bf16, device) into the tiled layout the LM
 * head streams fastest: tile (u, k) holds rows 64u..64u+63 and columns
 * 64k..64k+63, row-major; tiles ordered u-major, so the 64-row block of the
 * vocabulary that one work unit reads is one contiguous run of memory.
 * Rows and columns past the matrix are zero.  w_packed is a caller-owned
 * device buffer of ebd_lm_head_packed_bytes() bytes, 16-byte aligned.  A
 * one-time transform (model load); enqueued on stream. */
ebd_status ebd_pack_lm_head(ebd_handle* h, const uint16_t* w_lm, uint16_t* w_packed,
                            void* stream);

/* One EB decoding step (see top of file).  Enqueue only.  The kernels run
 * on `stream` in the order LM head, decision, window attention; the
 * attention (needed by neither of the others) may start while the decision
 * runs.  Later work on `stream` waits for all three. */
ebd_status ebd_step(ebd_handle* h, const ebd_step_args* a, void* stream);

/* Same step with the per-step tensors in HOST memory (pinned memory gives
 * asynchronous copies): cu_rows, prefix_len, row_pos, hidden, q, k_win,
 * v_win, tokens, mask, in_block, blk_meta and every non-NULL output are
 * host pointers; w_lm, k_cache and v_cache stay device pointers (resident
 * model weights and cache).  The handle copies the inputs to its own device
 * staging, runs the step and copies state and outputs back, all on
 * `stream`; the host buffers must stay valid until the stream reaches that
 * point (e.g. ebd_sync_status).  Enqueue only.
 * Pinned, mapped buffers (cudaHostAlloc / cudaHostRegister) move by kernel
 * instead of cudaMemcpyAsync.  With max_window <= 64 the kernels also write
 * the decode state and the outputs straight into such buffers (attn_out
 * when 16-byte aligned), and q, k_win and v_win come in on a copy engine on
 * the handle's own second stream while the LM head runs (the attention waits
 * for them, time-limited: EBD_ERR_TIMEOUT); `stream` waits for that stream
 * at the end of the step.  While `stream` is being captured into a CUDA
 * graph they go with the other inputs instead.  The state and outputs hold
 * the step's results only once the stream has passed the step, as in every
 * other case. */
ebd_status ebd_step_host(ebd_handle* h, const ebd_step_args* a, void* stream);

/* Only the decision (step 3) on caller-provided statistics: reads
 * a->conf, a->ent_norm, a->gap, a->argmax (device, [R]) as INPUTS, plus
 * cu_rows, row_pos and the decode state; writes the state, lbs_logit,
 * lps_prob and accepted.  hidden, q, k/v, w_lm and attn_out are ignored. */
ebd_status ebd_decide(ebd_handle* h, const ebd_step_args* a, void* stream);

/* Only step 2 (LM head + statistics) for a->rows rows of a->hidden:
 * writes conf, entropy, ent_norm, gap, argmax (any may be NULL). */
ebd_status ebd_lm_stats(ebd_handle* h, const ebd_step_args* a, void* stream);

/* ---- Vocabulary-parallel LM head (several GPUs) --------------------------
 * Step 2 sharded by vocabulary: GPU g holds rows [v_off_g, v_off_g +
 * v_count_g) of W_lm.  The statistics of App. B (Eq. app-confidence: kappa =
 * max_v p(v)), Sec. 5.1 (H~, x_hat) and Sec. 5.2 (Delta) are taken over the
 * whole vocabulary; the online-softmax state of a row over a vocabulary
 * range, (m = max logit, S = sum exp(l - m), T = sum exp(l - m)(l - m),
 * l2 = second largest logit, idx = lowest index of the maximum), merges
 * associatively, so each GPU reduces its range to one state per row, the
 * states are all-gathered (the caller's collective, e.g. NCCL), and every
 * GPU merges them into the statistics and runs the decision (ebd_decide)
 * on identical inputs.
 *
 * ebd_lm_shard_state: a->hidden and a->rows as for ebd_lm_stats; a->w_lm
 * points at this GPU's rows of W_lm (row-major [v_count][d_model], or the
 * tiled copy of those rows, which for v_off a multiple of 64 is the
 * contiguous slice of ebd_pack_lm_head's output starting at tile row
 * (v_off / 64) * ceil(d_model / 64) * 64); v_off must be a multiple of 64
 * and v_off + v_count <= vocab of the handle (the whole vocabulary).
 *   state  device float [a->rows][8], 16-byte aligned, caller-owned: per row
 *          m, S, T, l2, idx (int32 bits of a vocabulary index), 0, 0, 0.
 * ebd_merge_shard_states: states = device float [shards][a->rows][8] (the
 * gathered states, any shard order), 16-byte aligned; writes a->conf,
 * a->entropy, a->ent_norm, a->gap, a->argmax (any may be NULL), with
 * H~ = H / ln(vocab); a non-finite row records EBD_ERR_NONFINITE.
 * Both only enqueue on `stream`; argument errors return EBD_ERR_INVALID_ARG
 * and enqueue nothing. */
ebd_status ebd_lm_shard_state(ebd_handle* h, const ebd_step_args* a, int32_t v_off,
                              int32_t v_count, float* state, void* stream);
ebd_status ebd_merge_shard_states(ebd_handle* h, const float* states, int32_t shards,
                                  const ebd_step_args* a, void* stream);

/* Only step 1 (window attention): writes a->attn_out.  The handle picks one
 * of two kernels when it is created: the tcgen05 kernel (S and O in tensor
 * memory, one CTA per SM) for long key ranges or launches of few query
 * tiles, the mma.sync kernel (two CTAs per SM) for many tiles with short key
 * ranges; both compute the same attention.  The environment variables
 * EBD_ATTN_KERNEL = "tc" or "mma" and EBD_ATTN_SPLITS (key splits per query
 * tile, 1..8), read at ebd_create, override the choices. */
ebd_status ebd_attention(ebd_handle* h, const ebd_step_args* a, void* stream);

/* Synchronises `stream`, returns the first device-side failure recorded
 * since the last call (EBD_OK if none) and clears it. */
ebd_status ebd_sync_status(ebd_handle* h, void* stream);

/* Router weights as one bf16 blob, tensors row-major in this order:
 * LBS  ent1.w[64][1] ent1.b[64] ent2.w[64][64] ent2.b[64] ent_ln.g[64]
 *      ent_ln.b[64] tok.w[64][d_base] tok.b[64] comb.w[128][128] comb.b[128]
 *      pos[gen_len][128], then for l = 0, 1: qkv.w[384][128] qkv.b[384]
 *      out.w[128][128] out.b[128] ln1.g[128] ln1.b[128] ff1.w[256][128]
 *      ff1.b[256] ff2.w[128][256] ff2.b[128] ln2.g[128] ln2.b[128],
 *      head.w[1][128] head.b[1];
 * LPS  in.w[32][5] in.b[32] in_ln.g[32] in_ln.b[32], then for l = 0, 1:
 *      ln1.g[32] ln1.b[32] qkv.w[96][32] qkv.b[96] out.w[32][32] out.b[32]
 *      ln2.g[32] ln2.b[32] ff1.w[64][32] ff1.b[64] ff2.w[32][64] ff2.b[32],
 *      head.w[1][32] head.b[1].
 * (qkv rows: query, key, value blocks; head h uses rows h*dh..h*dh+dh-1 of
 * each block.)  With host == NULL only *bytes is set.  Synchronous. */
ebd_status ebd_export_weights(const ebd_handle* h, void* host, size_t* bytes);
ebd_status ebd_import_weights(ebd_handle* h, const void* host, size_t bytes);

/* The random init of ebd_create() computed on the host, without any CUDA
 * call: Linear weights and biases ~ U(-1/sqrt(fan_in), +1/sqrt(fan_in)),
 * LayerNorm gains 1 and biases 0, E_pos ~ U(-0.02*sqrt(3), +0.02*sqrt(3)),
 * from SplitMix64 used as a counter-based generator: with
 * G = 0x9E3779B97F4A7C15 and mix() the SplitMix64 output function,
 * key_t = mix(seed ^ ((t+1)*G)) for the t-th tensor of the blob order, and
 * element i draws u = (mix(key_t + (i+1)*G) >> 40) * 2^-24, then
 * w = bf16_rne((2u - 1) * bound) in float32.  With host == NULL only
 * *bytes is set. */
ebd_status ebd_router_init_host(const ebd_config* cfg, void* host, size_t* bytes);

/* Number of bf16 elements of the weight blob for cfg. */
size_t ebd_weight_count(const ebd_config* cfg);

/* Timing of ebd_step.  mode 0: off.  mode 1: every later ebd_step records
 * CUDA events on its stream around each kernel and runs them one after the
 * other (LM head, decision, window attention); ebd_profile_read writes the
 * durations in milliseconds to ms[0..2] = (attention, LM head, decision).
 * mode 2: the step runs as in production, the window attention overlapping
 * the decision; ms[1] = LM head, ms[2] = decision and attention together,
 * ms[0] = -1.  Events are recorded inside a captured graph too.
 * ebd_profile_read waits for the last recorded event; EBD_ERR_STATE if no
 * profiled step was recorded. */
ebd_status ebd_profile_enable(ebd_handle* h, int mode);
ebd_status ebd_profile_read(ebd_handle* h, float* ms);

/* Last error message of the handle (never NULL; "" if none). */
const char* ebd_last_error(const ebd_handle* h);

/* Library version string. */
const char* ebd_version(void);

/* Window of the next step of the generation loop (App. E algorithm in the
 * block-forward setting of Sec. 6.4; a host function, no device work).
 * Over the L response positions of one sequence with host arrays mask[L]
 * and in_block[L] and the block state meta[2] = {b, |B|} (|B| = 0: no
 * active block): f is the first masked position; with no active block the
 * window is [f, min(f + max_window, L)), with an active block [f, max B + 1)
 * where max B is the last position with in_block set.  Writes the window to
 * *lo, *hi (relative positions); *lo = *hi = L when no position is masked.
 * EBD_ERR_INVALID_ARG for a null pointer, L < 0 or max_window < 1;
 * EBD_ERR_STATE for an active block with no in_block position, or a window
 * longer than max_window. */
ebd_status ebd_loop_window(const uint8_t* mask, const uint8_t* in_block, const int32_t* meta,
                           int32_t L, int32_t max_window, int32_t* lo, int32_t* hi);

/* Window of the next step under the baselines' fixed blocks (App. B): the
 * first block [jB, jB + B) of the L response positions (host array mask[L])
 * that still holds a masked position, clipped to L.  *lo = *hi = L when none
 * does.  EBD_ERR_INVALID_ARG for a null pointer, L < 0 or block < 1.  A host
 * function, no device work. */
ebd_status ebd_loop_block_window(const uint8_t* mask, int32_t L, int32_t block, int32_t* lo,
                                 int32_t* hi);

/* ---- Allocation-free LM-head statistics ---------------------------------
 * No counterpart in the paper.  ebd_lm_stats_noalloc computes what
 * ebd_lm_stats computes (step 2: conf, entropy, ent_norm, gap, argmax of
 * `rows` rows of `hidden`, any output may be NULL), but takes no handle and
 * allocates no device memory, for callers that cannot allocate: a serving
 * process whose weight and KV-cache pools reserved the free HBM up front
 * (a further cudaMalloc fails or fragments them), or a decode loop that must
 * not stall on the device-wide synchronisation of cudaFree.
 *
 *   hidden   device, bf16 [rows][d_model], 16-byte aligned
 *   w_lm     device, bf16, 16-byte aligned: [vocab][d_model] row-major
 *            (w_lm_layout 0) or the tiled copy of ebd_pack_lm_head (1)
 *   rows     0 .. EBD_NOALLOC_MAX_ROWS; more returns EBD_ERR_UNSUPPORTED
 *   status   device int32 owned by the caller; it must be 0 before the
 *            call, and the kernels store the first device-side failure there
 *            (EBD_ERR_TIMEOUT, EBD_ERR_NONFINITE), as ebd_sync_status reports
 *            it for a handle
 *   stream   cudaStream_t as void*; the call only enqueues
 *
 * Scratch: the LM-head partials live in a statically sized device array of
 * EBD_NOALLOC_MAX_ROWS x EBD_NOALLOC_MAX_PARTS x 20 bytes (200 KiB), one per
 * device; nothing in it has to start at zero.  Calls that overlap in time on
 * one device (different streams or host threads) race on that array; calls
 * on one stream are ordered and safe.  The first call on each device does a
 * one-time setup (symbol address, kernel attributes) on the current device:
 * make that first call before any stream capture begins.
 * Returns EBD_ERR_INVALID_ARG for a null or misaligned pointer, a bad layout
 * or a size below its range, EBD_ERR_UNSUPPORTED beyond the maximum or on a
 * device other than sm_103, EBD_ERR_CUDA if a launch fails. */
#define EBD_NOALLOC_MAX_ROWS 64
#define EBD_NOALLOC_MAX_PARTS 160
ebd_status ebd_lm_stats_noalloc(const uint16_t* hidden, const uint16_t* w_lm,
                                int32_t w_lm_layout, int32_t rows, int32_t d_model,
                                int32_t vocab, float* conf, float* entropy, float* ent_norm,
                                float* gap, int32_t* argmax, int32_t* status, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* EBD_H_ */
