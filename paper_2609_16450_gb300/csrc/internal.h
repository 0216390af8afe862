// Launch parameters shared by the host side of the library and its kernels.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "ebd.h"
#include "lm_params.h"

namespace ebd {

// Checked builds (compiled with -DEBD_CHECKS): a global access whose index
// comes from device data (row offsets, positions, counts) is preceded by a
// check of the index against the buffer's extent; a failed check records
// EBD_ERR_BOUNDS in the status word and the access is skipped (nothing traps
// or waits).  In other builds the check compiles away.
__device__ __forceinline__ bool in_bounds(long long i, long long n, int* status) {
#ifdef EBD_CHECKS
  if (i >= 0 && i < n) return true;
  if (status != nullptr) atomicCAS(status, 0, EBD_ERR_BOUNDS);
  return false;
#else
  (void)i;
  (void)n;
  (void)status;
  return true;
#endif
}

constexpr int kMaxWindow = 64;        // window rows per sequence of the cluster decision
constexpr int kMaxSeqRows = 512;      // window rows per sequence of the grid-wide decision
constexpr int kUnit = 64;             // vocabulary rows per work unit of the LM head
constexpr int kLmThreads = 320;  // TMA warp, MMA warp, two epilogue warpgroups of 4 warps
constexpr int kMaxGroupRows = 512;    // rows per LM-head launch (TMEM: 512 columns)
constexpr int kDecideCluster = 8;     // CTAs per sequence in the decision kernel
constexpr int kDecideThreads = 256;
constexpr int kCtaWindow = 32;        // window rows per sequence of the one-CTA decision
constexpr int kCtaThreads = 512;
constexpr int kAttnThreads = 128;
constexpr int kAttnChunk = 64;        // keys per K/V tile
constexpr int kAttnStages = 3;
constexpr int kMaxAttnSplits = 8;
constexpr int kAttnTcThreads = 352;   // tcgen05 attention: K and V load warps, MMA warp, 8 softmax warps
constexpr int kAttnTcRows = 64;       // query rows per tile of the tcgen05 attention

// ------------------------------------------------------------------ attention
struct AttnParams {
  int B, Hq, Hkv, D, group;
  int R;                    // rows of the step (extent of q and out)
  int max_prefix;
  int max_qtiles, splits;
  int tc;                   // 1: the tcgen05 kernel, 0: the mma.sync kernel (64-row tiles)
  const int* cu_rows;
  const int* prefix_len;
  const int* suffix;        // [B][2] {s0, S} cached keys after the window, or null
  const __nv_bfloat16* q;   // [R][Hq][D]
  float* out;               // [R][Hq][D]
  float* part;              // [B*Hkv*max_qtiles*splits][tile rows][D] unnormalised O
  float* part_ml;           // [B*Hkv*max_qtiles*splits][tile rows][2] (max, sum) in log2 units
  int* tickets;             // [B*Hkv*max_qtiles]
  int* status;
  uint64_t limit_ns;
  int wait_prior;           // every CTA waits for the grid it depends on before exiting
  const unsigned* ready;     // non-null: q and the window K/V are being copied in by
  unsigned ready_ticket;    // another stream, which then writes ready_ticket to *ready
};

// ------------------------------------------------------------------ routers
// Device image of the router weights (layout in router_image.h).
struct RouterImage {
  const __nv_bfloat16* lbs_w;  // [8 ranks][LBS_W_ELEMS]
  const __nv_bfloat16* lps_w;  // [LPS_W_ELEMS]
  const float* vec;            // [8 ranks][V_ELEMS]
  const float* tok_table;      // [V][64] = W_tok W_e[v] (no bias)
  const __nv_bfloat16* cta_w;  // [rcta::kChunks][rcta::kChunkElems] (one-CTA kernel)
  const float* cta_vec;        // [rcta::S_ELEMS]
};

struct DecideParams {
  int B, V, grid_lm;        // grid_lm: LM-head partials per row
  int features_in;          // 1: conf/ent_norm/gap/argmax are inputs
  int pdl;                  // launched as a programmatic dependent of the LM head
  int warm;                 // one-CTA kernel: its CTAs find free SMs while the LM head
                            // runs, and each runs the decision once on a stand-in window
                            // before it waits for the LM head
  int mode, top_m;          // EBD_DECODE_*; commits per step of the Top-m rule
  int gen_len, g_max, l_min, l_b, eos_id, lps_enabled;
  float tau, tau_psi, inv_log_v;
  const int* cu_rows;
  const int* row_pos;
  const float4* part_f;
  const int* part_i;
  const int* tokens;         // decode state in: read before the LM head's grid completes
  const uint8_t* mask;
  const uint8_t* in_block;
  const int* blk_meta;
  int* tokens_out;           // decode state out: the same buffers as the state in,
  uint8_t* mask_out;         // unless the state in is a staged copy of the caller's
  uint8_t* in_block_out;
  int* blk_meta_out;
  float *conf, *entropy, *ent_norm, *gap, *lbs_logit, *lps_prob;
  int* argmax;
  uint8_t* accepted;
  int* status;
  int rows_expected;
  RouterImage w;
};

// ------------------------------------------------------------------ grid-wide decision
// fp32 copy of the router weights for the grid-wide decision (windows of up
// to kMaxSeqRows rows per sequence): float offsets into one allocation;
// matrices are stored [in][out] (consecutive outputs contiguous).
struct SeqLayer {                // one LBS encoder layer
  int qkv_t, qkv_b, out_t, out_b, ln1_g, ln1_b, ff1_t, ff1_b, ff2_t, ff2_b, ln2_g, ln2_b;
};
struct SeqBlock {                // one LPS block
  int ln1_g, ln1_b, qkv_t, qkv_b, out_t, out_b, ln2_g, ln2_b, ff1_t, ff1_b, ff2_t, ff2_b;
};
struct SeqWeights {
  int ent1_w, ent1_b, ent2_t, ent2_b, entln_g, entln_b, tok_b, comb_t, comb_b, pos;
  SeqLayer l[2];
  int head_w, head_b;
  int in_t, in_b, inln_g, inln_b;  // LPS input layer
  SeqBlock p[2];
  int phead_w, phead_b;
  int total;
};

struct SeqParams {
  int B, R, V, gen_len, g_max, l_min, l_b, eos_id, lps_enabled, mode, top_m;
  float tau, tau_psi;
  const int* cu_rows;
  const int* row_pos;
  int* tokens;
  uint8_t* mask;
  uint8_t* in_block;
  int* blk_meta;
  const float* conf;        // statistics of every row (inputs)
  const float* ent_norm;
  const float* gap;
  const int* argmax;
  uint8_t* accepted;        // outputs, may be null
  float* lbs_logit;
  float* lps_prob;
  const float* w;           // SeqWeights image
  SeqWeights o;
  const float* tok_table;   // [V][64]
  // scratch, [R] or [R][k] unless noted
  int* seq_of;
  int* mrank;               // rank of a masked row within its sequence's M, else -1
  int* mrows;               // sequence b's masked rows at [cu_rows[b], cu_rows[b] + |M|)
  int* bmrank;              // rank within B n M (rows the LPS scores), else -1
  int* bmrows;
  uint8_t* bad;
  uint8_t* ib;              // block membership after the selection
  int* sq;                  // [B + 1][8] per-sequence state (kSq* indices), then step flags
  float* O;                 // LBS logit
  float* P;                 // LPS probability
  float* feats;             // [R][8]
  float* Z;                 // [R][128]
  float* QKV;               // [R][384]
  float* A;                 // [R][128]
  float* Zp;                // [R][32]
  float* QKVp;              // [R][96]
  float* Ap;                // [R][32]
  int* status;
};

// host launchers (defined next to their kernels)
cudaError_t launch_lm_stats(const CUtensorMap& tmap_w, const CUtensorMap& tmap_h,
                            const LmParams& p, cudaStream_t st);
int lm_grid(int num_sms, int n_units);       // CTAs of the unpaired LM head
int lm_pair_grid(int num_sms, int n_units);  // CTAs of the paired (cta_group::2) LM head
// rows of an LM-head launch from which CTA pairs run it (and up to kMaxGroupRows)
constexpr int kLmPairMinRows = 65;
void lm_plan(LmParams& p, int rows, int V, int d, int num_sms, bool pair = false);
// pdl: launched as a programmatic dependent of the kernel before it on
// `st` (that kernel's CTAs release it early; the attention reads nothing the
// earlier kernel writes)
cudaError_t launch_attention(const CUtensorMap& kc, const CUtensorMap& vc, const CUtensorMap& kw,
                             const CUtensorMap& vw, const AttnParams& p, cudaStream_t st,
                             bool pdl = false);
cudaError_t launch_decide(const DecideParams& p, cudaStream_t st);
// the same decision with one CTA per sequence, for windows of up to
// kCtaWindow rows (k_decide_cta.cu)
cudaError_t launch_decide_cta(const DecideParams& p, cudaStream_t st);
// vocabulary-parallel LM head: one state per row from a launch's partials,
// and the statistics from the states of several shards (k_decide.cu)
cudaError_t launch_shard_state(const float4* part_f, const int* part_i, int rows, int grid,
                               float* state, cudaStream_t st);
cudaError_t launch_merge_shards(const float* states, int shards, int rows, int V, float inv_log_v,
                                float* conf, float* entropy, float* ent_norm, float* gap,
                                int* argmax, int* status, cudaStream_t st);
// the grid-wide decision: a chain of kernels on `st` (k_decide_seq.cu)
// the grid-wide decision: the scratch reset (before the LM head, so that the
// chain from the LM head on is unbroken), then the kernel chain; pdl_first:
// its first kernel is a programmatic dependent of the kernel before it
cudaError_t launch_decide_seq_init(const SeqParams& p, cudaStream_t st);
cudaError_t launch_decide_seq(const SeqParams& p, cudaStream_t st, bool pdl_first);
// prefix-cache append on commit: window row r of sequence b with mask[r] == 0
// is copied (K and V, Hkv * D bf16 each) to cache position row_pos[r] < Pmax
cudaError_t launch_kv_append(uint16_t* k_cache, uint16_t* v_cache, const uint16_t* k_win,
                             const uint16_t* v_win, const int* cu_rows, const int* row_pos,
                             const uint8_t* mask, int B, int rows, int Pmax, int hkvd,
                             cudaStream_t st, bool pdl);
cudaError_t launch_pack_lm(const __nv_bfloat16* w, __nv_bfloat16* out, int V, int d,
                           cudaStream_t st);
cudaError_t launch_fold_tok(const __nv_bfloat16* w_tok, const __nv_bfloat16* w_emb, float* table,
                            int V, int d_base, cudaStream_t st);

}  // namespace ebd
