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
//   embed     F_ent hidden and the token branch (warp per row); ent2 +
//             LayerNorm, fusion + E_pos (GEMMs)
//   2 layers  QKV (GEMM); attention (CTA per 8 queries and head, key blocks
//             staged in shared memory, one key per lane); output projection
//             + LayerNorm, FF1 + GELU, FF2 + LayerNorm (GEMMs); LBS head
//   select    candidates, MaxGapFilter, min-tokens fallback; B n M; LPS
//             features                                        (CTA per sequence)
//   LPS       input layer; 2 blocks as above (d 32, 4 heads); head, sigmoid
//   accept    union accept, anti-stall, commit, block resolution
// Products are fp32 FMAs on an fp32 copy of the (bf16-valued) weights stored
// [in][out].  The LBS products are CTA-tiled GEMMs over all window rows (8
// rows x 32*CPT columns per CTA, k-chunks staged in shared memory) with the
// bias, residual, LayerNorm, GELU or head fused into the epilogue: a warp
// holds one whole row of the tile.  Rows outside the LBS compute garbage in
// their own scratch rows, which nothing reads.  The small LPS products run
// one warp per row (a row's vector spread over the lanes, element lane + 32 i
// in register i, one input broadcast at a time) on the block's weights staged
// in shared memory.  Each kernel is a programmatic dependent of the one
// before it (seq_wait / seq_release below).
#include <climits>
#include <cstdlib>

#include "internal.h"

namespace ebd {

namespace {

constexpr int kSeqThreads = kMaxSeqRows;  // one thread per row in the per-sequence phases
constexpr int kWarpsPerCta = 8;
// per-sequence state, sq[b * 8 + k]
constexpr int kSqNM = 0, kSqRunLbs = 1, kSqNBM = 2, kSqMetaB = 3, kSqMetaS = 4, kSqRunLps = 5,
              kSqN = 6;
// step-wide flags after the per-sequence state: sq[8 * B + kFlagAnyLbs]
constexpr int kFlagAnyLbs = 0;

// Every kernel of the chain below is launched as a programmatic dependent of
// the one before it.  It waits for that grid's completion (and the
// visibility of its writes) before anything else (seq_wait), so each grid
// completes only after the one before it did.  The per-row and per-sequence
// kernels then let the next grid be scheduled at once (seq_release), which
// hides its launch behind their run; the LBS GEMM and attention kernels,
// which fill the SMs, release it only when they have no work (no LBS in the
// step), else by exiting: the next grid's waiting CTAs would take slots their
// own CTAs need (measured at 512 rows, step with the LBS / inside a block:
// releasing at entry everywhere 605 / 473 us, nowhere 582.5 / 482.5 us, as
// here 578 / 477 us).
__device__ __forceinline__ void seq_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void seq_release() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ float gelu_f(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}
__device__ __forceinline__ float wsum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
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

// The same with W and b in shared memory (plain loads).
template <int NI, int NO>
__device__ __forceinline__ void matvec_s(const float (&x)[NI], const float* W, const float* b,
                                         float (&y)[NO]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 0; o < NO; ++o) y[o] = b[lane + 32 * o];
#pragma unroll
  for (int i = 0; i < NI; ++i) {
#pragma unroll 8
    for (int kk = 0; kk < 32; ++kk) {
      const float xk = __shfl_sync(0xffffffffu, x[i], kk);
      const float* w = W + (32 * i + kk) * (32 * NO) + lane;
#pragma unroll
      for (int o = 0; o < NO; ++o) y[o] = fmaf(xk, w[32 * o], y[o]);
    }
  }
}

// Copies n floats of the weight image from offset `off` into shared memory
// (the whole CTA; the caller synchronises).
__device__ __forceinline__ void stage(float* dst, const float* __restrict__ w, int off, int n) {
  for (int i = threadIdx.x; i < n; i += blockDim.x) dst[i] = __ldg(w + off + i);
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
  seq_wait();
  seq_release();
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
    if (sq[kSqRunLbs]) atomicOr(p.sq + 8 * p.B + kFlagAnyLbs, 1);
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
// Multi-head attention of NQ query rows and one head over the rows
// `rows[0..n)`: softmax(q k^T / sqrt(DH)) v, qkv rows of stride LD with q at
// qo, k at ko, v at vo; query i is row qrows[i] (-1: none).  G = DH / 4 lanes
// share a key (4 dimensions each, one float4 of k and of v, loaded once for
// the NQ queries), so 32 / G keys are in flight per warp, each lane group
// with a running max and sum per query; the groups merge at the end.  Lanes
// [0, G) return, per query, the output dimensions 4 * lane .. 4 * lane + 3.
template <int DH, int NQ>
__device__ __forceinline__ void attend_rows(const float* __restrict__ qkv, int LD, const int (&qrows)[NQ],
                                            int qo, int ko, int vo, const int* __restrict__ rows,
                                            int n, float4 (&out)[NQ]) {
  constexpr int G = DH / 4, KP = 32 / G;
  const int lane = threadIdx.x & 31, grp = lane / G, sub = lane % G;
  const float scale = rsqrtf(static_cast<float>(DH));
  float4 q[NQ], o[NQ];
  float m[NQ], l[NQ];
#pragma unroll
  for (int i = 0; i < NQ; ++i) {
    q[i] = qrows[i] >= 0 ? *reinterpret_cast<const float4*>(qkv + static_cast<size_t>(qrows[i]) * LD + qo + 4 * sub)
                         : make_float4(0.f, 0.f, 0.f, 0.f);
    o[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    m[i] = -INFINITY;
    l[i] = 0.f;
  }
#pragma unroll 4
  for (int k0 = 0; k0 < n; k0 += KP) {
    const int k = k0 + grp;
    const bool ok = k < n;
    const float* kr = qkv + static_cast<size_t>(__ldg(rows + (ok ? k : 0))) * LD;
    const float4 kv = *reinterpret_cast<const float4*>(kr + ko + 4 * sub);
    const float4 vv = *reinterpret_cast<const float4*>(kr + vo + 4 * sub);
    float s[NQ];
#pragma unroll
    for (int i = 0; i < NQ; ++i) s[i] = q[i].x * kv.x + q[i].y * kv.y + q[i].z * kv.z + q[i].w * kv.w;
#pragma unroll
    for (int off = 1; off < G; off <<= 1)
#pragma unroll
      for (int i = 0; i < NQ; ++i) s[i] += __shfl_xor_sync(0xffffffffu, s[i], off);
#pragma unroll
    for (int i = 0; i < NQ; ++i) {
      const float si = ok ? s[i] * scale : -INFINITY;
      const float mn = fmaxf(m[i], si);
      const float c = mn == -INFINITY ? 1.f : expf(m[i] - mn), e = mn == -INFINITY ? 0.f : expf(si - mn);
      l[i] = l[i] * c + e;
      o[i].x = fmaf(e, vv.x, o[i].x * c);
      o[i].y = fmaf(e, vv.y, o[i].y * c);
      o[i].z = fmaf(e, vv.z, o[i].z * c);
      o[i].w = fmaf(e, vv.w, o[i].w * c);
      m[i] = mn;
    }
  }
#pragma unroll
  for (int i = 0; i < NQ; ++i) {
    float M = m[i];
#pragma unroll
    for (int off = G; off < 32; off <<= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    const float c = m[i] == -INFINITY ? 0.f : expf(m[i] - M);
    float li = l[i] * c;
    float4 oi = make_float4(o[i].x * c, o[i].y * c, o[i].z * c, o[i].w * c);
#pragma unroll
    for (int off = G; off < 32; off <<= 1) {
      li += __shfl_xor_sync(0xffffffffu, li, off);
      oi.x += __shfl_xor_sync(0xffffffffu, oi.x, off);
      oi.y += __shfl_xor_sync(0xffffffffu, oi.y, off);
      oi.z += __shfl_xor_sync(0xffffffffu, oi.z, off);
      oi.w += __shfl_xor_sync(0xffffffffu, oi.w, off);
    }
    const float il = 1.0f / li;
    out[i] = make_float4(oi.x * il, oi.y * il, oi.z * il, oi.w * il);
  }
}

// Tiled fp32 GEMM over the window rows: CTA (blockIdx.x, blockIdx.y)
// computes rows [8 bx, 8 bx + 8) x columns [32 CPT by, +32 CPT) of
// A[R][lda] (first K columns) times W[K][ldw]; warp w owns row 8 bx + w,
// lane l columns l + 32 j (j < CPT).  K is staged in chunks of kGemmK rows,
// double-buffered: the next chunk's global loads are in flight while the
// current one is multiplied.  epi(row, acc[CPT], col0) gets a warp's row
// (rows >= R included: their A rows read as zero).
constexpr int kGemmK = 32;  // k-chunk staged per step
constexpr int kGemmRows = 8;
template <int CPT, class Epi>
__device__ __forceinline__ void gemm_rows(const float* __restrict__ A, int lda, int K,
                                          const float* __restrict__ W, int ldw, int R, Epi epi) {
  constexpr int NC = 32 * CPT;
  constexpr int NB4 = kGemmK * NC / 4 / 256;  // float4 of a B chunk per thread
  static_assert(NB4 * 256 * 4 == kGemmK * NC, "B chunk split");
  static_assert(kGemmRows * kGemmK == 256, "one A element per thread");
  __shared__ __align__(16) float As[2][kGemmRows][kGemmK];
  __shared__ __align__(16) float Bs[2][kGemmK][NC];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int row0 = blockIdx.x * kGemmRows, col0 = blockIdx.y * NC;
  const int ar = tid / kGemmK, ak = tid % kGemmK;  // this thread's A element of a chunk
  const bool arow = row0 + ar < R;
  float acc[CPT];
#pragma unroll
  for (int j = 0; j < CPT; ++j) acc[j] = 0.f;
  float ra;
  float4 rb[NB4];
  auto load = [&](int k0) {
    ra = arow ? A[static_cast<size_t>(row0 + ar) * lda + k0 + ak] : 0.f;
#pragma unroll
    for (int u = 0; u < NB4; ++u) {
      const int it = tid + 256 * u, kk = it / (NC / 4), c4 = it % (NC / 4);
      rb[u] = __ldg(reinterpret_cast<const float4*>(W + static_cast<size_t>(k0 + kk) * ldw + col0 + 4 * c4));
    }
  };
  auto store = [&](int buf) {
    As[buf][ar][ak] = ra;
#pragma unroll
    for (int u = 0; u < NB4; ++u) {
      const int it = tid + 256 * u, kk = it / (NC / 4), c4 = it % (NC / 4);
      *reinterpret_cast<float4*>(&Bs[buf][kk][4 * c4]) = rb[u];
    }
  };
  load(0);
  store(0);
  __syncthreads();
  const int nch = K / kGemmK;
  for (int c = 0; c < nch; ++c) {
    const int buf = c & 1;
    if (c + 1 < nch) load((c + 1) * kGemmK);
#pragma unroll 8
    for (int kk = 0; kk < kGemmK; ++kk) {
      const float a = As[buf][warp][kk];
#pragma unroll
      for (int j = 0; j < CPT; ++j) acc[j] = fmaf(a, Bs[buf][kk][lane + 32 * j], acc[j]);
    }
    if (c + 1 < nch) store(buf ^ 1);
    __syncthreads();
  }
  epi(row0 + warp, acc, col0);
}

__device__ __forceinline__ bool any_lbs(const SeqParams& p) {
  return p.sq[8 * p.B + kFlagAnyLbs] != 0;
}

// F_ent hidden (Linear 1 -> 64, GELU) of H~ -> U[r][0..64), and the token
// branch W_tok W_e[x_hat] + b (folded table) -> X[r][64..128)  (Eq. lbs_feat)
__global__ void __launch_bounds__(256) lbs_pre_kernel(const SeqParams p) {
  seq_wait();
  seq_release();
  const int lane = threadIdx.x & 31;
  const int r = lbs_row(p, blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5));
  if (r < 0) return;
  const float* w = p.w;
  const float h = p.ent_norm[r];
  const int tok = p.argmax[r];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int c = lane + 32 * i;
    p.A[static_cast<size_t>(r) * 128 + c] = gelu_f(fmaf(w[p.o.ent1_w + c], h, w[p.o.ent1_b + c]));
    p.Z[static_cast<size_t>(r) * 128 + 64 + c] =
        (tok >= 0 && tok < p.V ? __ldg(p.tok_table + static_cast<size_t>(tok) * 64 + c) : 0.f) +
        w[p.o.tok_b + c];
  }
}

// e = LN(W_ent2 u + b) -> X[r][0..64)  (X lives in Z; U in A)
__global__ void __launch_bounds__(256) lbs_ent2_kernel(const SeqParams p) {
  seq_wait();
  if (!any_lbs(p)) {
    seq_release();
    return;
  }
  const float* w = p.w;
  gemm_rows<2>(p.A, 128, 64, w + p.o.ent2_t, 64, p.R, [&](int r, float (&acc)[2], int) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < 2; ++j) acc[j] += w[p.o.ent2_b + lane + 32 * j];
    layer_norm_w<2>(acc, w + p.o.entln_g, w + p.o.entln_b);
    if (r < p.R)
#pragma unroll
      for (int j = 0; j < 2; ++j) p.Z[static_cast<size_t>(r) * 128 + lane + 32 * j] = acc[j];
  });
}

// z = W_combine [e; t] + b + E_pos[rank], in place in Z: a CTA owns all 128
// columns of its rows and has read them before its epilogue
__global__ void __launch_bounds__(256) lbs_comb_kernel(const SeqParams p) {
  seq_wait();
  if (!any_lbs(p)) {
    seq_release();
    return;
  }
  const float* w = p.w;
  gemm_rows<4>(p.Z, 128, 128, w + p.o.comb_t, 128, p.R, [&](int r, float (&acc)[4], int) {
    const int lane = threadIdx.x & 31;
    if (r >= p.R) return;
    const int k = p.mrank[r];
    const float* pos = w + p.o.pos + static_cast<size_t>(k < 0 ? 0 : k) * 128;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      p.Z[static_cast<size_t>(r) * 128 + lane + 32 * j] =
          acc[j] + w[p.o.comb_b + lane + 32 * j] + pos[lane + 32 * j];
  });
}

__global__ void __launch_bounds__(256) lbs_qkv_kernel(const SeqParams p, int l) {
  seq_wait();
  if (!any_lbs(p)) {
    seq_release();
    return;
  }
  const SeqLayer& L = p.o.l[l];
  const float* bq = p.w + L.qkv_b;
  gemm_rows<1>(p.Z, 128, 128, p.w + L.qkv_t, 384, p.R, [&](int r, float (&acc)[1], int col0) {
    const int lane = threadIdx.x & 31;
    if (r < p.R) p.QKV[static_cast<size_t>(r) * 384 + col0 + lane] = acc[0] + bq[col0 + lane];
  });
}

// LBS attention: CTA (x, h, b) takes 8 queries of sequence b's M (rank
// 8 x + w for warp w) and head h (32 dimensions).  Blocks of 64 keys (k and
// v of head h) are staged in shared memory once for the 8 warps,
// double-buffered (the next block's loads are in flight while the current
// one is used), rows padded to 33 floats so that 32 lanes reading 32
// different rows hit 32 banks.  Each lane of a warp takes whole keys: the
// full 32-dimension score, then its own running max, sum and output row
// (no shuffles per key).  At the end the lanes' states are merged: the
// common max, then a reduce-scatter of the 32 output dimensions that leaves
// dimension d in lane d.
constexpr int kAttnKB = 64;
constexpr int kAttnLd = 33;
__global__ void __launch_bounds__(256) lbs_attn_kernel(const SeqParams p) {
  seq_wait();
  __shared__ float Ks[2][kAttnKB][kAttnLd];
  __shared__ float Vs[2][kAttnKB][kAttnLd];
  static_assert(kAttnKB * 16 == 4 * 256, "four float4 of a key block per thread");
  const int b = blockIdx.z, h = blockIdx.y, qb = blockIdx.x;
  const int* sq = p.sq + 8 * b;
  const int nM = sq[kSqNM];
  if (!sq[kSqRunLbs] || qb * 8 >= nM) {  // uniform over the CTA
    seq_release();
    return;
  }
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int* rows = p.mrows + p.cu_rows[b];
  const int qi = qb * 8 + warp;
  const int qr = qi < nM ? rows[qi] : -1;
  float q[32], o[32];
  {
    const float* qp = p.QKV + static_cast<size_t>(qr >= 0 ? qr : rows[0]) * 384 + 32 * h;
    const float scale = rsqrtf(32.0f);
#pragma unroll
    for (int d4 = 0; d4 < 8; ++d4) {
      const float4 v = *reinterpret_cast<const float4*>(qp + 4 * d4);
      q[4 * d4 + 0] = v.x * scale;
      q[4 * d4 + 1] = v.y * scale;
      q[4 * d4 + 2] = v.z * scale;
      q[4 * d4 + 3] = v.w * scale;
    }
  }
#pragma unroll
  for (int d = 0; d < 32; ++d) o[d] = 0.f;
  float m = -INFINITY, l = 0.f;
  float4 pre[4];
  auto fetch = [&](int kb) {  // item it: key it / 16, float4 it % 8 of k (it % 16 < 8) or v
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int it = tid + 256 * u, key = it >> 4, part = it & 15, c4 = part & 7;
      const int kidx = kb + key;
      pre[u] = kidx < nM ? *reinterpret_cast<const float4*>(p.QKV + static_cast<size_t>(rows[kidx]) * 384 +
                                                            (part < 8 ? 128 : 256) + 32 * h + 4 * c4)
                         : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  };
  auto put = [&](int buf) {
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int it = tid + 256 * u, key = it >> 4, part = it & 15, c4 = part & 7;
      float* dst = part < 8 ? &Ks[buf][key][4 * c4] : &Vs[buf][key][4 * c4];
      dst[0] = pre[u].x;
      dst[1] = pre[u].y;
      dst[2] = pre[u].z;
      dst[3] = pre[u].w;
    }
  };
  fetch(0);
  put(0);
  __syncthreads();
  for (int kb = 0, buf = 0; kb < nM; kb += kAttnKB, buf ^= 1) {
    const bool more = kb + kAttnKB < nM;
    if (more) fetch(kb + kAttnKB);
    const int nk = min(kAttnKB, nM - kb);
#pragma unroll 1
    for (int k0 = 0; k0 < nk; k0 += 32) {
      const int k = k0 + lane;
      if (k < nk) {
        const float* kr = Ks[buf][k];
        float s = 0.f;
#pragma unroll
        for (int d = 0; d < 32; ++d) s = fmaf(q[d], kr[d], s);
        const float mn = fmaxf(m, s);
        const float c = expf(m - mn), e = expf(s - mn);  // m = -inf first: c = 0
        l = fmaf(l, c, e);
        const float* vr = Vs[buf][k];
#pragma unroll
        for (int d = 0; d < 32; ++d) o[d] = fmaf(e, vr[d], o[d] * c);
        m = mn;
      }
    }
    if (more) put(buf ^ 1);  // the buffer every warp finished with before the last barrier
    __syncthreads();
  }
  // merge the 32 lanes: common max, then sums; lanes that saw no key hold
  // m = -inf and contribute nothing
  float M = m;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  const float c = m == -INFINITY ? 0.f : expf(m - M);
  l *= c;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
#pragma unroll
  for (int d = 0; d < 32; ++d) o[d] *= c;
  // reduce-scatter: at offset `off` a lane keeps the half of its live
  // values selected by (lane & off) and adds its partner's copy of it
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const bool up = (lane & off) != 0;
#pragma unroll
    for (int i = 0; i < off; ++i) {
      const float give = up ? o[i] : o[i + off];
      const float keep = up ? o[i + off] : o[i];
      o[i] = keep + __shfl_xor_sync(0xffffffffu, give, off);
    }
  }
  if (qr >= 0) p.A[static_cast<size_t>(qr) * 128 + 32 * h + lane] = o[0] / l;
}

// z = LN1(z + W_out a + b), in place (post-norm layer)
__global__ void __launch_bounds__(256) lbs_out_kernel(const SeqParams p, int l) {
  seq_wait();
  if (!any_lbs(p)) {
    seq_release();
    return;
  }
  const SeqLayer& L = p.o.l[l];
  const float* w = p.w;
  gemm_rows<4>(p.A, 128, 128, w + L.out_t, 128, p.R, [&](int r, float (&acc)[4], int) {
    const int lane = threadIdx.x & 31;
    const int rr = r < p.R ? r : 0;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      acc[j] += w[L.out_b + lane + 32 * j] + p.Z[static_cast<size_t>(rr) * 128 + lane + 32 * j];
    layer_norm_w<4>(acc, w + L.ln1_g, w + L.ln1_b);
    if (r < p.R)
#pragma unroll
      for (int j = 0; j < 4; ++j) p.Z[static_cast<size_t>(r) * 128 + lane + 32 * j] = acc[j];
  });
}

// h = GELU(W_1 z + b_1) -> the QKV scratch (256 of its 384 columns)
__global__ void __launch_bounds__(256) lbs_ff1_kernel(const SeqParams p, int l) {
  seq_wait();
  if (!any_lbs(p)) {
    seq_release();
    return;
  }
  const SeqLayer& L = p.o.l[l];
  const float* b1 = p.w + L.ff1_b;
  gemm_rows<1>(p.Z, 128, 128, p.w + L.ff1_t, 256, p.R, [&](int r, float (&acc)[1], int col0) {
    const int lane = threadIdx.x & 31;
    if (r < p.R) p.QKV[static_cast<size_t>(r) * 384 + col0 + lane] = gelu_f(acc[0] + b1[col0 + lane]);
  });
}

// z = LN2(z + W_2 h + b_2), in place; after the last layer the LBS head
// O = w . z + b
__global__ void __launch_bounds__(256) lbs_ff2_kernel(const SeqParams p, int l) {
  seq_wait();
  if (!any_lbs(p)) {
    seq_release();
    return;
  }
  const SeqLayer& L = p.o.l[l];
  const float* w = p.w;
  gemm_rows<4>(p.QKV, 384, 256, w + L.ff2_t, 128, p.R, [&](int r, float (&acc)[4], int) {
    const int lane = threadIdx.x & 31;
    const int rr = r < p.R ? r : 0;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      acc[j] += w[L.ff2_b + lane + 32 * j] + p.Z[static_cast<size_t>(rr) * 128 + lane + 32 * j];
    layer_norm_w<4>(acc, w + L.ln2_g, w + L.ln2_b);
    if (r >= p.R) return;
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      p.Z[static_cast<size_t>(r) * 128 + lane + 32 * j] = acc[j];
      s = fmaf(acc[j], w[p.o.head_w + lane + 32 * j], s);
    }
    if (l == 1) {
      s = wsum(s) + w[p.o.head_b];
      if (lane == 0 && lbs_row(p, r) >= 0) p.O[r] = s;
    }
  });
}

// ------------------------------------------------------------------ selection
// B of each sequence (App. E algorithm, block selection; Readings R8, R9),
// then B n M in ascending position and the LPS features (Reading R13)
__global__ void __launch_bounds__(kSeqThreads) seq_select_kernel(const SeqParams p) {
  seq_wait();
  seq_release();
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
  seq_wait();
  seq_release();
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

// pre-norm block: LN1 and QKV.  The LPS kernels run one warp per row of
// B n M; a CTA with any such row stages the block's weights in shared
// memory first (a few KB, read once from L2 instead of once per row).
__global__ void __launch_bounds__(256) lps_qkv_kernel(const SeqParams p, int l) {
  seq_wait();
  seq_release();
  __shared__ float s_ln[64], s_qkv[32 * 96], s_qkvb[96];
  const int lane = threadIdx.x & 31;
  const int r = lps_row(p, blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5));
  if (!__syncthreads_or(r >= 0)) return;  // uniform over the CTA
  const SeqBlock& L = p.o.p[l];
  stage(s_ln, p.w, L.ln1_g, 32);
  stage(s_ln + 32, p.w, L.ln1_b, 32);
  stage(s_qkv, p.w, L.qkv_t, 32 * 96);
  stage(s_qkvb, p.w, L.qkv_b, 96);
  __syncthreads();
  if (r < 0) return;
  float y[1] = {p.Zp[static_cast<size_t>(r) * 32 + lane]}, q[3];
  layer_norm_w<1>(y, s_ln, s_ln + 32);
  matvec_s<1, 3>(y, s_qkv, s_qkvb, q);
#pragma unroll
  for (int i = 0; i < 3; ++i) p.QKVp[static_cast<size_t>(r) * 96 + lane + 32 * i] = q[i];
}

__global__ void __launch_bounds__(256) lps_attn_kernel(const SeqParams p) {
  seq_wait();
  seq_release();
  const int lane = threadIdx.x & 31;
  const int wid = blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  const int r = lps_row(p, wid >> 2), h = wid & 3;
  if (r < 0) return;
  const int b = p.seq_of[r];
  const int q[1] = {r};
  float4 v[1];
  attend_rows<8, 1>(p.QKVp, 96, q, 8 * h, 32 + 8 * h, 64 + 8 * h, p.bmrows + p.cu_rows[b],
                    p.sq[8 * b + kSqNBM], v);
  if (lane < 2) *reinterpret_cast<float4*>(p.Ap + static_cast<size_t>(r) * 32 + 8 * h + 4 * lane) = v[0];
}

// output projection + residual, LN2, FFN + residual; after the last block
// the head and p_psi = sigmoid(O_psi)
__global__ void __launch_bounds__(256) lps_out_ffn_kernel(const SeqParams p, int l) {
  seq_wait();
  seq_release();
  __shared__ float s_out[32 * 32], s_ff1[32 * 64], s_ff2[64 * 32], s_vec[32 * 4 + 64];
  const int lane = threadIdx.x & 31;
  const int r = lps_row(p, blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5));
  if (!__syncthreads_or(r >= 0)) return;  // uniform over the CTA
  const SeqBlock& L = p.o.p[l];
  const float* w = p.w;
  float* s_outb = s_vec;
  float* s_ln2 = s_vec + 32;  // gamma, beta
  float* s_ff2b = s_vec + 96;
  float* s_ff1b = s_vec + 128;
  stage(s_out, w, L.out_t, 32 * 32);
  stage(s_ff1, w, L.ff1_t, 32 * 64);
  stage(s_ff2, w, L.ff2_t, 64 * 32);
  stage(s_outb, w, L.out_b, 32);
  stage(s_ln2, w, L.ln2_g, 32);
  stage(s_ln2 + 32, w, L.ln2_b, 32);
  stage(s_ff2b, w, L.ff2_b, 32);
  stage(s_ff1b, w, L.ff1_b, 64);
  __syncthreads();
  if (r < 0) return;
  float a[1] = {p.Ap[static_cast<size_t>(r) * 32 + lane]}, y[1], z = p.Zp[static_cast<size_t>(r) * 32 + lane];
  matvec_s<1, 1>(a, s_out, s_outb, y);
  z += y[0];
  float t[1] = {z}, hdn[2], f[1];
  layer_norm_w<1>(t, s_ln2, s_ln2 + 32);
  matvec_s<1, 2>(t, s_ff1, s_ff1b, hdn);
  hdn[0] = gelu_f(hdn[0]);
  hdn[1] = gelu_f(hdn[1]);
  matvec_s<2, 1>(hdn, s_ff2, s_ff2b, f);
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
  seq_wait();
  seq_release();
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
  if (acc && in_bounds(r, p.R, p.status)) {
    p.tokens[r] = p.argmax[r];
    msk = false;
  }
  const bool inb = row && p.ib[r] != 0;
  if (inb && msk) atomicOr(&s_open, 1);
  __syncthreads();
  const bool resolve = p.mode == EBD_DECODE_EB && meta_s > 0 && !s_open;
  if (row && in_bounds(r, p.R, p.status)) {
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

namespace {
template <typename... KArgs, typename... Args>
cudaError_t chain(void (*k)(KArgs...), dim3 grid, dim3 block, cudaStream_t st, bool pdl, Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, k, args...);
}
}  // namespace

cudaError_t launch_decide_seq_init(const SeqParams& p, cudaStream_t st) {
  if (p.B <= 0 || p.R <= 0) return cudaSuccess;
  cudaError_t e;
  if ((e = cudaMemsetAsync(p.mrank, 0xff, static_cast<size_t>(p.R) * sizeof(int), st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(p.bmrank, 0xff, static_cast<size_t>(p.R) * sizeof(int), st)) != cudaSuccess) return e;
  return cudaMemsetAsync(p.sq + 8 * p.B, 0, 8 * sizeof(int), st);
}

cudaError_t launch_decide_seq(const SeqParams& p, cudaStream_t st, bool pdl_first) {
  if (p.B <= 0 || p.R <= 0) return cudaSuccess;
  const unsigned rows_grid = static_cast<unsigned>((p.R + kWarpsPerCta - 1) / kWarpsPerCta);
  const unsigned head_grid = static_cast<unsigned>((4 * p.R + kWarpsPerCta - 1) / kWarpsPerCta);
  const dim3 t256(256), tseq(kSeqThreads);
  cudaError_t e = chain(seq_prep_kernel, dim3(p.B), tseq, st, pdl_first, p);
  auto add = [&](cudaError_t x) {
    if (e == cudaSuccess) e = x;
  };
  if (p.mode == EBD_DECODE_EB) {
    const unsigned tiles = static_cast<unsigned>((p.R + kGemmRows - 1) / kGemmRows);
    const dim3 attn_grid(kMaxSeqRows / 8, 4, static_cast<unsigned>(p.B));
    add(chain(lbs_pre_kernel, dim3(rows_grid), t256, st, true, p));
    add(chain(lbs_ent2_kernel, dim3(tiles, 1), t256, st, true, p));
    add(chain(lbs_comb_kernel, dim3(tiles, 1), t256, st, true, p));
    for (int l = 0; l < 2; ++l) {
      add(chain(lbs_qkv_kernel, dim3(tiles, 12), t256, st, true, p, l));
      add(chain(lbs_attn_kernel, attn_grid, t256, st, true, p));
      add(chain(lbs_out_kernel, dim3(tiles, 1), t256, st, true, p, l));
      add(chain(lbs_ff1_kernel, dim3(tiles, 8), t256, st, true, p, l));
      add(chain(lbs_ff2_kernel, dim3(tiles, 1), t256, st, true, p, l));
    }
  }
  add(chain(seq_select_kernel, dim3(p.B), tseq, st, true, p));
  if (p.mode == EBD_DECODE_EB && p.lps_enabled) {
    add(chain(lps_in_kernel, dim3(rows_grid), t256, st, true, p));
    for (int l = 0; l < 2; ++l) {
      add(chain(lps_qkv_kernel, dim3(rows_grid), t256, st, true, p, l));
      add(chain(lps_attn_kernel, dim3(head_grid), t256, st, true, p));
      add(chain(lps_out_ffn_kernel, dim3(rows_grid), t256, st, true, p, l));
    }
  }
  add(chain(seq_accept_kernel, dim3(p.B), tseq, st, true, p));
  return e;
}

}  // namespace ebd
