// The EB decision for windows of up to kMaxSeqRows (512) rows per sequence:
// the full-sequence setting, where every position of the response is a row
// of the step (App. E algorithm "Inference with LBS Block Selection and LPS
// Parallel Commit" with M = all masked positions of the response; LBS,
// Sec. 5.1 and App. C.1; LPS, Sec. 5.2 and App. D.1; baseline rules, App. B
// Eq. prelim-update).
//
// The cluster decision keeps a sequence's LBS activations in shared memory,
// which holds 64 rows.  Here every phase is a grid-wide kernel over the rows
// of all sequences, with the activations in an L2-resident scratch:
//   prep      masked set M of each sequence (compaction), LBS on/off
//   embed     F_ent and the token branch, fusion + E_pos      (warp per row)
//   2 layers  QKV; attention (warp per row and head); output projection,
//             LayerNorm, FFN, LayerNorm (warp per row); LBS head
//   select    candidates, MaxGapFilter, min-tokens fallback; B n M; LPS
//             features                                        (CTA per sequence)
//   LPS       input layer; 2 blocks as above (d 32, 4 heads); head, sigmoid
//   accept    union accept, anti-stall, commit, block resolution
// Products are fp32 FMAs on an fp32 copy of the (bf16-valued) weights stored
// [in][out]: a warp holds a row's vector spread over its lanes (element
// lane + 32 i in register i) and broadcasts one input at a time.
#include <climits>

#include "internal.h"

namespace ebd {

namespace {

constexpr int kSeqThreads = kMaxSeqRows;  // one thread per row in the per-sequence phases
constexpr int kWarpsPerCta = 8;
// per-sequence state, sq[b * 8 + k]
constexpr int kSqNM = 0, kSqRunLbs = 1, kSqNBM = 2, kSqMetaB = 3, kSqMetaS = 4, kSqRunLps = 5,
              kSqN = 6;

__device__ __forceinline__ float gelu_f(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}
__device__ __forceinline__ float wsum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float wmax(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// y = W^T x + b: x has KI = 32 * NI inputs (lane holds x[lane + 32 i] in
// x[i]), W is [KI][32 * NO], y has 32 * NO outputs laid out the same way.
template <int NI, int NO>
__device__ __forceinline__ void matvec(const float (&x)[NI], const float* __restrict__ W,
                                       const float* __restrict__ b, float (&y)[NO]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 0; o < NO; ++o) y[o] = b[lane + 32 * o];
#pragma unroll
  for (int i = 0; i < NI; ++i) {
#pragma unroll 4
    for (int kk = 0; kk < 32; ++kk) {
      const float xk = __shfl_sync(0xffffffffu, x[i], kk);
      const float* w = W + static_cast<size_t>(32 * i + kk) * (32 * NO) + lane;
#pragma unroll
      for (int o = 0; o < NO; ++o) y[o] = fmaf(xk, __ldg(w + 32 * o), y[o]);
    }
  }
}

// LayerNorm (eps 1e-5) of a warp-spread vector of 32 * N values
template <int N>
__device__ __forceinline__ void layer_norm_w(float (&v)[N], const float* __restrict__ g,
                                             const float* __restrict__ b) {
  const int lane = threadIdx.x & 31;
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < N; ++i) s += v[i];
  const float mean = wsum(s) * (1.0f / (32 * N));
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < N; ++i) q += (v[i] - mean) * (v[i] - mean);
  const float inv = 1.0f / sqrtf(wsum(q) * (1.0f / (32 * N)) + 1e-5f);
#pragma unroll
  for (int i = 0; i < N; ++i) v[i] = (v[i] - mean) * inv * g[lane + 32 * i] + b[lane + 32 * i];
}

// Block-wide exclusive scan of a 0/1 flag over the kSeqThreads threads;
// returns the flag's rank and writes the total to *total (all threads).
__device__ __forceinline__ int block_rank(bool flag, int* warp_tot, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t bal = __ballot_sync(0xffffffffu, flag);
  if (lane == 0) warp_tot[warp] = __popc(bal);
  __syncthreads();
  int base = 0, tot = 0;
  for (int w = 0; w < (kSeqThreads >> 5); ++w) {
    if (w < warp) base += warp_tot[w];
    tot += warp_tot[w];
  }
  __syncthreads();
  *total = tot;
  return base + __popc(bal & ((1u << lane) - 1u));
}

// ------------------------------------------------------------------ prep
__global__ void __launch_bounds__(kSeqThreads) seq_prep_kernel(const SeqParams p) {
  __shared__ int warp_tot[kSeqThreads / 32];
  const int b = blockIdx.x, j = threadIdx.x;
  const int r0 = p.cu_rows[b], r1 = p.cu_rows[b + 1];
  int n = r1 - r0;
  if (n < 0 || n > kMaxSeqRows || r0 < 0 || r1 > p.R || n > p.gen_len) {
    if (j == 0) atomicCAS(p.status, 0, EBD_ERR_INVALID_ARG);
    n = 0;
  }
  const int r = r0 + j;
  bool m = false;
  if (j < n) {
    const float c = p.conf[r], e = p.ent_norm[r], g = p.gap[r];
    const int a = p.argmax[r];
    const bool bad = !(isfinite(c) && isfinite(e) && isfinite(g)) || a < 0 || a >= p.V;
    p.bad[r] = bad ? 1 : 0;
    p.seq_of[r] = b;
    p.O[r] = __int_as_float(0x7fc00000);
    p.P[r] = __int_as_float(0x7fc00000);
    m = p.mask[r] != 0;
  }
  int nM;
  const int k = block_rank(m, warp_tot, &nM);
  if (j < n) {
    p.mrank[r] = m ? k : -1;
    p.bmrank[r] = -1;
    if (m) p.mrows[r0 + k] = r;
  }
  if (j == 0) {
    int* sq = p.sq + 8 * b;
    const int meta_s = p.blk_meta[2 * b + 1];
    sq[kSqNM] = nM;
    sq[kSqRunLbs] = (p.mode == EBD_DECODE_EB && meta_s == 0 && nM > p.l_min) ? 1 : 0;
    sq[kSqNBM] = 0;
    sq[kSqMetaB] = p.blk_meta[2 * b];
    sq[kSqMetaS] = meta_s;
    sq[kSqRunLps] = 0;
    sq[kSqN] = n;
  }
}

// the row of this warp if the LBS runs for it (masked, its sequence runs
// the LBS), else -1
__device__ __forceinline__ int lbs_row(const SeqParams& p, int r) {
  if (r >= p.R || p.mrank[r] < 0) return -1;
  return p.sq[8 * p.seq_of[r] + kSqRunLbs] ? r : -1;
}
__device__ __forceinline__ int lps_row(const SeqParams& p, int r) {
  if (r >= p.R || p.bmrank[r] < 0) return -1;
  return p.sq[8 * p.seq_of[r] + kSqRunLps] ? r : -1;
}

// ------------------------------------------------------------------ LBS
// F_ent (Linear 1->64, GELU, Linear 64->64, LayerNorm) of H~, the token
// branch W_tok W_e[x_hat] + b (folded table), fusion W_combine [e; t] + b +
// E_pos[rank]  (Eq. lbs_feat)
__global__ void __launch_bounds__(256) lbs_embed_kernel(const SeqParams p) {
  const int lane = threadIdx.x & 31;
  const int r = lbs_row(p, blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5));
  if (r < 0) return;
  const float* w = p.w;
  const float h = p.ent_norm[r];
  float u[2], e[2];
#pragma unroll
  for (int i = 0; i < 2; ++i)
    u[i] = gelu_f(fmaf(w[p.o.ent1_w + lane + 32 * i], h, w[p.o.ent1_b + lane + 32 * i]));
  matvec<2, 2>(u, w + p.o.ent2_t, w + p.o.ent2_b, e);
  layer_norm_w<2>(e, w + p.o.entln_g, w + p.o.entln_b);
  const int tok = p.argmax[r];
  float x[4] = {e[0], e[1], 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < 2; ++i)
    x[2 + i] = (tok >= 0 && tok < p.V ? __ldg(p.tok_table + static_cast<size_t>(tok) * 64 + lane + 32 * i) : 0.f) +
               w[p.o.tok_b + lane + 32 * i];
  float z[4];
  matvec<4, 4>(x, w + p.o.comb_t, w + p.o.comb_b, z);
  const float* pos = w + p.o.pos + static_cast<size_t>(p.mrank[r]) * 128;
#pragma unroll
  for (int i = 0; i < 4; ++i) p.Z[static_cast<size_t>(r) * 128 + lane + 32 * i] = z[i] + pos[lane + 32 * i];
}

__global__ void __launch_bounds__(256) lbs_qkv_kernel(const SeqParams p, int l) {
  const int lane = threadIdx.x & 31;
  const int r = lbs_row(p, blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5));
  if (r < 0) return;
  const SeqLayer& L = p.o.l[l];
  float z[4], y[12];
#pragma unroll
  for (int i = 0; i < 4; ++i) z[i] = p.Z[static_cast<size_t>(r) * 128 + lane + 32 * i];
  matvec<4, 12>(z, p.w + L.qkv_t, p.w + L.qkv_b, y);
#pragma unroll
  for (int i = 0; i < 12; ++i) p.QKV[static_cast<size_t>(r) * 384 + lane + 32 * i] = y[i];
}

// softmax(q k^T / sqrt(DH)) v of one row and one head over the rows of
// `rows[0..n)`; qkv rows of stride LD with q at qo, k at ko, v at vo.  The
// lanes split the keys (running max and sum each), then merge.  Returns the
// output element `lane` (lanes >= DH return 0).
template <int DH>
__device__ __forceinline__ float attend_row(const float* __restrict__ qkv, int LD, int r, int qo,
                                            int ko, int vo, const int* __restrict__ rows, int n) {
  const int lane = threadIdx.x & 31;
  float q[DH], o[DH];
  const float* qp = qkv + static_cast<size_t>(r) * LD + qo;
#pragma unroll
  for (int d = 0; d < DH; ++d) {
    q[d] = qp[d];
    o[d] = 0.f;
  }
  const float scale = rsqrtf(static_cast<float>(DH));
  float m = -INFINITY, l = 0.f;
  for (int k = lane; k < n; k += 32) {
    const float* kr = qkv + static_cast<size_t>(rows[k]) * LD;
    float s = 0.f;
#pragma unroll
    for (int d = 0; d < DH; ++d) s = fmaf(q[d], kr[ko + d], s);
    s *= scale;
    const float mn = fmaxf(m, s);
    const float c = expf(m - mn), e = expf(s - mn);
    l = l * c + e;
#pragma unroll
    for (int d = 0; d < DH; ++d) o[d] = fmaf(e, kr[vo + d], o[d] * c);
    m = mn;
  }
  const float M = wmax(m);
  const float c = m == -INFINITY ? 0.f : expf(m - M);
  const float L = wsum(l * c);
  float mine = 0.f;
#pragma unroll
  for (int d = 0; d < DH; ++d) {
    const float t = wsum(o[d] * c);
    if (d == lane) mine = t;
  }
  return mine / L;
}

__global__ void __launch_bounds__(256) lbs_attn_kernel(const SeqParams p) {
  const int lane = threadIdx.x & 31;
  const int wid = blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  const int r = lbs_row(p, wid >> 2), h = wid & 3;
  if (r < 0) return;
  const int b = p.seq_of[r];
  const float v = attend_row<32>(p.QKV, 384, r, 32 * h, 128 + 32 * h, 256 + 32 * h,
                                 p.mrows + p.cu_rows[b], p.sq[8 * b + kSqNM]);
  p.A[static_cast<size_t>(r) * 128 + 32 * h + lane] = v;
}

// output projection + residual + LN1, FFN + residual + LN2 (post-norm
// layer); after the last layer, the LBS head O = w . z + b
__global__ void __launch_bounds__(256) lbs_out_ffn_kernel(const SeqParams p, int l) {
  const int lane = threadIdx.x & 31;
  const int r = lbs_row(p, blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5));
  if (r < 0) return;
  const SeqLayer& L = p.o.l[l];
  const float* w = p.w;
  float a[4], z[4], y[4], hdn[8], f[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    a[i] = p.A[static_cast<size_t>(r) * 128 + lane + 32 * i];
    z[i] = p.Z[static_cast<size_t>(r) * 128 + lane + 32 * i];
  }
  matvec<4, 4>(a, w + L.out_t, w + L.out_b, y);
#pragma unroll
  for (int i = 0; i < 4; ++i) z[i] += y[i];
  layer_norm_w<4>(z, w + L.ln1_g, w + L.ln1_b);
  matvec<4, 8>(z, w + L.ff1_t, w + L.ff1_b, hdn);
#pragma unroll
  for (int i = 0; i < 8; ++i) hdn[i] = gelu_f(hdn[i]);
  matvec<8, 4>(hdn, w + L.ff2_t, w + L.ff2_b, f);
#pragma unroll
  for (int i = 0; i < 4; ++i) z[i] += f[i];
  layer_norm_w<4>(z, w + L.ln2_g, w + L.ln2_b);
#pragma unroll
  for (int i = 0; i < 4; ++i) p.Z[static_cast<size_t>(r) * 128 + lane + 32 * i] = z[i];
  if (l == 1) {
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) s = fmaf(z[i], w[p.o.head_w + lane + 32 * i], s);
    s = wsum(s) + w[p.o.head_b];
    if (lane == 0) p.O[r] = s;
  }
}

// ------------------------------------------------------------------ selection
// B of each sequence (App. E algorithm, block selection; Readings R8, R9),
// then B n M in ascending position and the LPS features (Reading R13)
__global__ void __launch_bounds__(kSeqThreads) seq_select_kernel(const SeqParams p) {
  __shared__ int warp_tot[kSeqThreads / 32];
  __shared__ int cpos[kMaxSeqRows];
  __shared__ int s_cut, s_first;
  const int b = blockIdx.x, j = threadIdx.x;
  int* sq = p.sq + 8 * b;
  const int n = sq[kSqN], nM = sq[kSqNM];
  const int r0 = p.cu_rows[b], r = r0 + j;
  int meta_b = sq[kSqMetaB], meta_s = sq[kSqMetaS];
  const bool row = j < n;
  const bool m = row && p.mask[r] != 0;
  const bool bad = row && p.bad[r] != 0;
  const int pos = row ? p.row_pos[r] : 0;
  bool inb = row && p.in_block[r] != 0;
  if (p.mode != EBD_DECODE_EB) {
    inb = row;  // the window is the active fixed block; no block state
  } else if (meta_s == 0) {
    bool sel;
    int nB;
    if (nM <= p.l_min) {
      sel = m;
      nB = nM;
    } else {
      const bool cand = m && p.O[r] > 0.f && p.argmax[r] != p.eos_id && !bad;
      int nC;
      const int c = block_rank(cand, warp_tot, &nC);
      if (cand) cpos[c] = pos;
      if (j == 0) s_cut = nC;
      __syncthreads();
      // MaxGapFilter: cut at the first candidate farther than g_max from its predecessor
      if (cand && c >= 1 && cpos[c] - cpos[c - 1] > p.g_max) atomicMin(&s_cut, c);
      __syncthreads();
      nB = s_cut;
      sel = cand && c < nB;
      if (nB < p.l_min) {  // min-tokens fallback: the first min(L_B, |M|) masked rows
        nB = nM < p.l_b ? nM : p.l_b;
        sel = m && p.mrank[r] < nB;
      }
    }
    inb = sel;
    if (j == 0) s_first = INT_MAX;
    __syncthreads();
    if (sel) atomicMin(&s_first, j);
    __syncthreads();
    if (nB > 0) {
      meta_b = p.row_pos[r0 + s_first];
      meta_s = nB;
    }
  }
  if (row) p.ib[r] = inb ? 1 : 0;
  const bool bm = inb && m && !bad;
  int nBM;
  const int k = block_rank(bm, warp_tot, &nBM);
  if (bm) {
    p.bmrank[r] = k;
    p.bmrows[r0 + k] = r;
    if (p.mode == EBD_DECODE_EB && meta_s > 0) {
      float* f = p.feats + static_cast<size_t>(r) * 8;
      f[0] = p.conf[r];
      f[1] = p.ent_norm[r];
      f[2] = p.gap[r];
      f[3] = static_cast<float>(nBM) / static_cast<float>(meta_s);
      f[4] = static_cast<float>(pos - meta_b) / static_cast<float>(meta_s);
    }
  }
  if (j == 0) {
    sq[kSqNBM] = nBM;
    sq[kSqMetaB] = meta_b;
    sq[kSqMetaS] = meta_s;
    sq[kSqRunLps] = (p.mode == EBD_DECODE_EB && p.lps_enabled && nBM > 0) ? 1 : 0;
  }
}

// ------------------------------------------------------------------ LPS
// Linear(5 -> 32), LayerNorm, GELU
__global__ void __launch_bounds__(256) lps_in_kernel(const SeqParams p) {
  const int lane = threadIdx.x & 31;
  const int r = lps_row(p, blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5));
  if (r < 0) return;
  const float* w = p.w;
  const float* f = p.feats + static_cast<size_t>(r) * 8;
  float y[1] = {w[p.o.in_b + lane]};
#pragma unroll
  for (int k = 0; k < 5; ++k) y[0] = fmaf(f[k], w[p.o.in_t + k * 32 + lane], y[0]);
  layer_norm_w<1>(y, w + p.o.inln_g, w + p.o.inln_b);
  p.Zp[static_cast<size_t>(r) * 32 + lane] = gelu_f(y[0]);
}

// pre-norm block: LN1 and QKV
__global__ void __launch_bounds__(256) lps_qkv_kernel(const SeqParams p, int l) {
  const int lane = threadIdx.x & 31;
  const int r = lps_row(p, blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5));
  if (r < 0) return;
  const SeqBlock& L = p.o.p[l];
  float y[1] = {p.Zp[static_cast<size_t>(r) * 32 + lane]}, q[3];
  layer_norm_w<1>(y, p.w + L.ln1_g, p.w + L.ln1_b);
  matvec<1, 3>(y, p.w + L.qkv_t, p.w + L.qkv_b, q);
#pragma unroll
  for (int i = 0; i < 3; ++i) p.QKVp[static_cast<size_t>(r) * 96 + lane + 32 * i] = q[i];
}

__global__ void __launch_bounds__(256) lps_attn_kernel(const SeqParams p) {
  const int lane = threadIdx.x & 31;
  const int wid = blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  const int r = lps_row(p, wid >> 2), h = wid & 3;
  if (r < 0) return;
  const int b = p.seq_of[r];
  const float v = attend_row<8>(p.QKVp, 96, r, 8 * h, 32 + 8 * h, 64 + 8 * h,
                                p.bmrows + p.cu_rows[b], p.sq[8 * b + kSqNBM]);
  if (lane < 8) p.Ap[static_cast<size_t>(r) * 32 + 8 * h + lane] = v;
}

// output projection + residual, LN2, FFN + residual; after the last block
// the head and p_psi = sigmoid(O_psi)
__global__ void __launch_bounds__(256) lps_out_ffn_kernel(const SeqParams p, int l) {
  const int lane = threadIdx.x & 31;
  const int r = lps_row(p, blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5));
  if (r < 0) return;
  const SeqBlock& L = p.o.p[l];
  const float* w = p.w;
  float a[1] = {p.Ap[static_cast<size_t>(r) * 32 + lane]}, y[1], z = p.Zp[static_cast<size_t>(r) * 32 + lane];
  matvec<1, 1>(a, w + L.out_t, w + L.out_b, y);
  z += y[0];
  float t[1] = {z}, hdn[2], f[1];
  layer_norm_w<1>(t, w + L.ln2_g, w + L.ln2_b);
  matvec<1, 2>(t, w + L.ff1_t, w + L.ff1_b, hdn);
  hdn[0] = gelu_f(hdn[0]);
  hdn[1] = gelu_f(hdn[1]);
  matvec<2, 1>(hdn, w + L.ff2_t, w + L.ff2_b, f);
  z += f[0];
  p.Zp[static_cast<size_t>(r) * 32 + lane] = z;
  if (l == 1) {
    const float o = wsum(z * w[p.o.phead_w + lane]) + w[p.o.phead_b];
    if (lane == 0) p.P[r] = 1.0f / (1.0f + expf(-o));
  }
}

// ------------------------------------------------------------------ accept
// union accept (Reading R14), anti-stall fallback, parallel commit, block
// resolution; the baselines' rules (Reading R20) in their modes
__global__ void __launch_bounds__(kSeqThreads) seq_accept_kernel(const SeqParams p) {
  __shared__ float s_conf[kMaxSeqRows];
  __shared__ int s_pos[kMaxSeqRows];
  __shared__ int s_any, s_best, s_open;
  const int b = blockIdx.x, j = threadIdx.x;
  int* sq = p.sq + 8 * b;
  const int n = sq[kSqN], nBM = sq[kSqNBM];
  int meta_b = sq[kSqMetaB], meta_s = sq[kSqMetaS];
  const int r0 = p.cu_rows[b], r = r0 + j;
  const bool row = j < n;
  const int k = row ? p.bmrank[r] : -1;
  const bool bm = k >= 0;
  const float conf = row ? p.conf[r] : 0.f;
  const int pos = row ? p.row_pos[r] : 0;
  if (bm) {
    s_conf[k] = conf;
    s_pos[k] = pos;
  }
  if (j == 0) {
    s_any = 0;
    s_best = -1;
    s_open = 0;
  }
  __syncthreads();
  bool acc = false;
  if (bm) {
    if (p.mode == EBD_DECODE_TOPM) {
      int rank = 0;  // rows ahead: higher kappa, or equal kappa and lower position
      for (int i = 0; i < nBM; ++i)
        rank += (s_conf[i] > conf || (s_conf[i] == conf && s_pos[i] < pos)) ? 1 : 0;
      acc = rank < p.top_m;
    } else {
      acc = conf >= p.tau ||
            (p.mode == EBD_DECODE_EB && p.lps_enabled && p.P[r] > p.tau_psi);
    }
    if (acc) atomicOr(&s_any, 1);
  }
  __syncthreads();
  if (!s_any && nBM > 0) {  // anti-stall: the highest kappa, lowest position on ties
    if (bm) {
      bool best = true;
      for (int i = 0; i < nBM; ++i)
        if (s_conf[i] > conf || (s_conf[i] == conf && s_pos[i] < pos)) best = false;
      if (best) s_best = k;
    }
    __syncthreads();
    acc = bm && k == s_best;
  }
  bool msk = row && p.mask[r] != 0;
  if (acc) {
    p.tokens[r] = p.argmax[r];
    msk = false;
  }
  const bool inb = row && p.ib[r] != 0;
  if (inb && msk) atomicOr(&s_open, 1);
  __syncthreads();
  const bool resolve = p.mode == EBD_DECODE_EB && meta_s > 0 && !s_open;
  if (row) {
    p.mask[r] = msk ? 1 : 0;
    if (p.mode == EBD_DECODE_EB) p.in_block[r] = (inb && !resolve) ? 1 : 0;
    if (p.accepted) p.accepted[r] = acc ? 1 : 0;
    if (p.lbs_logit) p.lbs_logit[r] = p.O[r];
    if (p.lps_prob) p.lps_prob[r] = p.P[r];
  }
  if (j == 0 && p.mode == EBD_DECODE_EB) {
    if (resolve) meta_b = meta_s = 0;
    p.blk_meta[2 * b] = meta_b;
    p.blk_meta[2 * b + 1] = meta_s;
  }
}

}  // namespace

cudaError_t launch_decide_seq(const SeqParams& p, cudaStream_t st) {
  if (p.B <= 0 || p.R <= 0) return cudaSuccess;
  cudaError_t e;
  if ((e = cudaMemsetAsync(p.mrank, 0xff, static_cast<size_t>(p.R) * sizeof(int), st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(p.bmrank, 0xff, static_cast<size_t>(p.R) * sizeof(int), st)) != cudaSuccess) return e;
  const unsigned rows_grid = static_cast<unsigned>((p.R + kWarpsPerCta - 1) / kWarpsPerCta);
  const unsigned head_grid = static_cast<unsigned>((4 * p.R + kWarpsPerCta - 1) / kWarpsPerCta);
  seq_prep_kernel<<<p.B, kSeqThreads, 0, st>>>(p);
  if (p.mode == EBD_DECODE_EB) {
    lbs_embed_kernel<<<rows_grid, 256, 0, st>>>(p);
    for (int l = 0; l < 2; ++l) {
      lbs_qkv_kernel<<<rows_grid, 256, 0, st>>>(p, l);
      lbs_attn_kernel<<<head_grid, 256, 0, st>>>(p);
      lbs_out_ffn_kernel<<<rows_grid, 256, 0, st>>>(p, l);
    }
  }
  seq_select_kernel<<<p.B, kSeqThreads, 0, st>>>(p);
  if (p.mode == EBD_DECODE_EB && p.lps_enabled) {
    lps_in_kernel<<<rows_grid, 256, 0, st>>>(p);
    for (int l = 0; l < 2; ++l) {
      lps_qkv_kernel<<<rows_grid, 256, 0, st>>>(p, l);
      lps_attn_kernel<<<head_grid, 256, 0, st>>>(p);
      lps_out_ffn_kernel<<<rows_grid, 256, 0, st>>>(p, l);
    }
  }
  seq_accept_kernel<<<p.B, kSeqThreads, 0, st>>>(p);
  return cudaGetLastError();
}

}  // namespace ebd
