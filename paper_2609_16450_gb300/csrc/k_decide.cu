// The EB decision for every sequence of a step (App. E, algorithm
// "Inference with LBS Block Selection and LPS Parallel Commit"):
//   1. merge the LM-head partial states of each window row into
//      kappa, H, H~ = H / ln|V|, Delta and x_hat (App. B, Sec. 5.1, Sec. 5.2);
//   2. with no active block and |M| > L_min: the LBS router (Sec. 5.1,
//      App. C.1) over the masked rows, then EOS removal, MaxGapFilter and the
//      min-tokens fallback; with |M| <= L_min: B = M;
//   3. the LPS router (Sec. 5.2, App. D.1) over the masked rows of B with
//      features (kappa, H~, Delta, rho, pos);
//   4. union accept, anti-stall fallback, parallel commit, block resolution.
//
// One thread-block cluster of 8 CTAs per sequence.  The LBS encoder is split
// across the cluster by output features (and, for attention, by head and
// query half); every CTA keeps a full copy of the activations and the
// slices are exchanged through distributed shared memory.  Router matmuls
// are fp32 FMA on bf16-stored weights.  The LPS router and the decision run
// in rank 0.
#include <cooperative_groups.h>

#include <climits>

#include "internal.h"
#include "ptx.cuh"
#include "router_image.h"

namespace cg = cooperative_groups;

namespace ebd {

namespace {

using namespace rimg;

constexpr int W = kMaxWindow;  // rows per sequence
constexpr int LDZ = 132;       // residual stream / [e;t] / attention concat
constexpr int LDKV = 68;       // k in [0,32), v in [32,64)
constexpr int LDQ = 36;
constexpr int LDS = 68;
// activation pool (floats), LBS phase
constexpr int P_Z = 0;                  // [64][132] residual stream z
constexpr int P_X = P_Z + W * LDZ;      // [64][132] [e;t] | concat | FFN partial inbox [8][64][16]
constexpr int P_KV = P_X + W * LDZ;     // [64][68]  k,v of this CTA's head | FFN hidden [64][36]
constexpr int P_Q = P_KV + W * LDKV;    // [32][36]  queries of this CTA's half
constexpr int P_S = P_Q + 32 * LDQ;     // [32][68]  attention scores
constexpr int POOL = P_S + 32 * LDS;    // 24576 floats
// activation pool, LPS phase (rank 0)
constexpr int L_Z = 0, L_Y = 2304, L_F = 4608, L_QKV = 5120, L_ATT = 11520, L_SC = 13824,
              L_H = 18176;
static_assert(L_H + W * 68 <= POOL, "LPS pool layout");
static_assert(8 * W * 16 <= W * LDZ, "FFN partial inbox");

struct __align__(16) Smem {
  __nv_bfloat16 w[LBS_W_ELEMS];   // this rank's LBS weight slices
  __nv_bfloat16 lw[LPS_W_ELEMS];  // LPS weights (rank 0)
  float v[V_ELEMS];               // vectors
  float pool[POOL];
  float f_conf[W], f_ent[W], f_gap[W], f_O[W], f_p[W];
  int f_arg[W], f_pos[W], f_tok[W], Mrows[W], Brows[W], BMrows[W];
  uint8_t f_mask[W], f_ib[W], f_acc[W], f_bad[W];
  int nM, nBM, meta_b, meta_s, n_rows, r0, run_lbs, bad_seq, wait_fail;
  uint64_t bar;
};

__device__ __forceinline__ float gelu(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ void bulk_copy(void* smem_dst, const void* gsrc, uint32_t bytes,
                                          uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(smem_dst)),
      "l"(gsrc), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// out(j, o) = bias[o] + sum_k in[j][k] * Wt[k][o] for j < n, o < Os (Os even);
// Wt is shared-memory bf16 [K][ldw].  epi(j, o, value) consumes the result.
template <class Epi>
__device__ __forceinline__ void gemm_rows(const float* in, int ldi, int n, int K,
                                          const __nv_bfloat16* Wt, int ldw, int Os,
                                          const float* bias, Epi epi) {
  const int pairs = Os >> 1;
  const int ldw2 = ldw >> 1;
  for (int it = threadIdx.x; it < n * pairs; it += blockDim.x) {
    const int j = it / pairs, pr = it - j * pairs;
    float a0 = bias ? bias[2 * pr] : 0.f, a1 = bias ? bias[2 * pr + 1] : 0.f;
    const float* x = in + j * ldi;
    const __nv_bfloat162* w = reinterpret_cast<const __nv_bfloat162*>(Wt) + pr;
    int k = 0;
#pragma unroll 2
    for (; k + 4 <= K; k += 4) {
      const float4 xv = *reinterpret_cast<const float4*>(x + k);
      const float2 w0 = __bfloat1622float2(w[(k + 0) * ldw2]);
      const float2 w1 = __bfloat1622float2(w[(k + 1) * ldw2]);
      const float2 w2 = __bfloat1622float2(w[(k + 2) * ldw2]);
      const float2 w3 = __bfloat1622float2(w[(k + 3) * ldw2]);
      a0 = fmaf(xv.x, w0.x, a0); a1 = fmaf(xv.x, w0.y, a1);
      a0 = fmaf(xv.y, w1.x, a0); a1 = fmaf(xv.y, w1.y, a1);
      a0 = fmaf(xv.z, w2.x, a0); a1 = fmaf(xv.z, w2.y, a1);
      a0 = fmaf(xv.w, w3.x, a0); a1 = fmaf(xv.w, w3.y, a1);
    }
    for (; k < K; ++k) {
      const float2 wk = __bfloat1622float2(w[k * ldw2]);
      a0 = fmaf(x[k], wk.x, a0);
      a1 = fmaf(x[k], wk.y, a1);
    }
    epi(j, 2 * pr, a0);
    epi(j, 2 * pr + 1, a1);
  }
}

// LayerNorm (eps 1e-5) over `dim` (32, 64 or 128) of rows j < n; warp per row.
__device__ __forceinline__ void layer_norm_rows(const float* src, int lds, float* dst, int ldd,
                                                int n, int dim, const float* g, const float* b) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = blockDim.x >> 5;
  const int per = dim >> 5;
  for (int j = warp; j < n; j += nw) {
    float v[4] = {0.f, 0.f, 0.f, 0.f};
    float s = 0.f;
    for (int c = 0; c < per; ++c) {
      v[c] = src[j * lds + lane + 32 * c];
      s += v[c];
    }
    const float mean = warp_sum(s) / dim;
    float q = 0.f;
    for (int c = 0; c < per; ++c) {
      const float d = v[c] - mean;
      q += d * d;
    }
    const float inv = 1.0f / sqrtf(warp_sum(q) / dim + 1e-5f);
    for (int c = 0; c < per; ++c) {
      const int o = lane + 32 * c;
      dst[j * ldd + o] = (v[c] - mean) * inv * g[o] + b[o];
    }
  }
}

// Scaled dot-product attention of queries qs[i] (i < nq) over keys/values
// k < n (head width dh); writes o(i, d) through epi.  S: [nq][LDS] scratch.
template <class Epi>
__device__ __forceinline__ void attend(const float* qs, int ldq, const float* ks, const float* vs,
                                       int ldkv, int nq, int n, int dh, float* S, Epi epi) {
  const float scale = 1.0f / sqrtf(static_cast<float>(dh));
  for (int it = threadIdx.x; it < nq * n; it += blockDim.x) {
    const int i = it / n, k = it - i * n;
    float a = 0.f;
    for (int d = 0; d < dh; ++d) a = fmaf(qs[i * ldq + d], ks[k * ldkv + d], a);
    S[i * LDS + k] = a * scale;
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = warp; i < nq; i += (blockDim.x >> 5)) {
    const float x0 = lane < n ? S[i * LDS + lane] : -INFINITY;
    const float x1 = lane + 32 < n ? S[i * LDS + lane + 32] : -INFINITY;
    const float m = warp_max(fmaxf(x0, x1));
    const float e0 = lane < n ? expf(x0 - m) : 0.f;
    const float e1 = lane + 32 < n ? expf(x1 - m) : 0.f;
    const float inv = 1.0f / warp_sum(e0 + e1);
    if (lane < n) S[i * LDS + lane] = e0 * inv;
    if (lane + 32 < n) S[i * LDS + lane + 32] = e1 * inv;
  }
  __syncthreads();
  for (int it = threadIdx.x; it < nq * dh; it += blockDim.x) {
    const int i = it / dh, d = it - i * dh;
    float a = 0.f;
    for (int k = 0; k < n; ++k) a = fmaf(S[i * LDS + k], vs[k * ldkv + d], a);
    epi(i, d, a);
  }
}

__device__ __forceinline__ void merge_state(float& m, float& s, float& t, float& l2, int& idx,
                                            float bm, float bs, float bt, float bl2, int bidx) {
  if (bm > m || (bm == m && bidx < idx)) {
    float x;
    int xi;
    x = m; m = bm; bm = x;
    x = s; s = bs; bs = x;
    x = t; t = bt; bt = x;
    x = l2; l2 = bl2; bl2 = x;
    xi = idx; idx = bidx; bidx = xi;
  }
  l2 = fmaxf(l2, bm);
  if (bm == -INFINITY) return;
  const float dl = bm - m;
  const float sc = expf(dl);
  t = t + sc * (bt + dl * bs);
  s = s + sc * bs;
}

// ----------------------------------------------------------------- LPS (rank 0)
// Sec. 5.2 / App. D.1: Linear(5->32) -> LayerNorm -> GELU, two pre-norm blocks
// (4 heads, FFN 64, GELU), head Linear(32->1); p_psi = sigmoid(O).
__device__ void lps_forward(Smem& sm, int n) {
  float* P = sm.pool;
  float* zL = P + L_Z;
  float* yL = P + L_Y;
  float* fL = P + L_F;
  float* qkv = P + L_QKV;
  float* att = P + L_ATT;
  float* sc = P + L_SC;
  float* h64 = P + L_H;
  const float* V = sm.v + V_LPS;
  constexpr int LD = 36, LDQKV = 100;
  const float rho = static_cast<float>(sm.nBM) / static_cast<float>(sm.meta_s);
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    const int r = sm.BMrows[i];
    fL[i * 8 + 0] = sm.f_conf[r];
    fL[i * 8 + 1] = sm.f_ent[r];
    fL[i * 8 + 2] = sm.f_gap[r];
    fL[i * 8 + 3] = rho;
    fL[i * 8 + 4] = static_cast<float>(sm.f_pos[r] - sm.meta_b) / static_cast<float>(sm.meta_s);
  }
  __syncthreads();
  for (int it = threadIdx.x; it < n * 32; it += blockDim.x) {
    const int i = it >> 5, o = it & 31;
    float a = V[VP_INB + o];
    for (int k = 0; k < 5; ++k) a = fmaf(fL[i * 8 + k], V[VP_INT + k * 32 + o], a);
    yL[i * LD + o] = a;
  }
  __syncthreads();
  layer_norm_rows(yL, LD, zL, LD, n, 32, V + VP_INLNG, V + VP_INLNB);
  __syncthreads();
  for (int it = threadIdx.x; it < n * 32; it += blockDim.x) {
    const int i = it >> 5, o = it & 31;
    zL[i * LD + o] = gelu(zL[i * LD + o]);
  }
  __syncthreads();
  for (int l = 0; l < 2; ++l) {
    const __nv_bfloat16* Wl = sm.lw + l * PL_STRIDE;
    const float* Vl = V + VP_LAYER0 + l * VP_LAYER_STRIDE;
    layer_norm_rows(zL, LD, yL, LD, n, 32, Vl + VPL_LN1G, Vl + VPL_LN1B);
    __syncthreads();
    gemm_rows(yL, LD, n, 32, Wl + PL_QKV, 96, 96, Vl + VPL_QKVB,
              [&](int j, int o, float v) { qkv[j * LDQKV + o] = v; });
    __syncthreads();
    for (int h = 0; h < 4; ++h) {
      attend(qkv + 8 * h, LDQKV, qkv + 32 + 8 * h, qkv + 64 + 8 * h, LDQKV, n, n, 8, sc,
             [&](int i, int d, float v) { att[i * LD + 8 * h + d] = v; });
      __syncthreads();
    }
    gemm_rows(att, LD, n, 32, Wl + PL_OUT, 32, 32, Vl + VPL_OUTB,
              [&](int j, int o, float v) { zL[j * LD + o] += v; });
    __syncthreads();
    layer_norm_rows(zL, LD, yL, LD, n, 32, Vl + VPL_LN2G, Vl + VPL_LN2B);
    __syncthreads();
    gemm_rows(yL, LD, n, 32, Wl + PL_FF1, 64, 64, Vl + VPL_FF1B,
              [&](int j, int o, float v) { h64[j * 68 + o] = gelu(v); });
    __syncthreads();
    gemm_rows(h64, 68, n, 64, Wl + PL_FF2, 32, 32, Vl + VPL_FF2B,
              [&](int j, int o, float v) { zL[j * LD + o] += v; });
    __syncthreads();
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = warp; i < n; i += (blockDim.x >> 5)) {
    const float a = warp_sum(zL[i * LD + lane] * V[VP_HEADW + lane]) + V[VP_HEADB];
    if (lane == 0) sm.f_p[sm.BMrows[i]] = 1.0f / (1.0f + expf(-a));
  }
  __syncthreads();
}

}  // namespace

__global__ void __cluster_dims__(kDecideCluster, 1, 1) __launch_bounds__(kDecideThreads, 1)
    decide_kernel(const DecideParams p) {
  extern __shared__ uint8_t smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 15) & ~static_cast<uintptr_t>(15));
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int seq = blockIdx.x / kDecideCluster;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  float* const P = sm.pool;

  if (tid == 0) {
    // weights and vectors of this rank: bulk copies issued first, so they
    // land while the statistics are merged
    mbar_init(&sm.bar, 1);
    fence_mbar_init();
    const uint32_t wb = LBS_W_ELEMS * 2u, lb = LPS_W_ELEMS * 2u, vb = V_ELEMS * 4u;
    mbar_arrive_expect_tx(&sm.bar, wb + vb + (rank == 0 ? lb : 0u));
    bulk_copy(sm.w, p.w.lbs_w + static_cast<size_t>(rank) * LBS_W_ELEMS, wb, &sm.bar);
    bulk_copy(sm.v, p.w.vec + static_cast<size_t>(rank) * V_ELEMS, vb, &sm.bar);
    if (rank == 0) bulk_copy(sm.lw, p.w.lps_w, lb, &sm.bar);
    const int r0 = p.cu_rows[seq], r1 = p.cu_rows[seq + 1];
    const int n = r1 - r0;
    sm.bad_seq = 0;
    if (p.cu_rows[p.B] != p.rows_expected || n < 0 || n > W || r0 < 0) {
      sm.bad_seq = 1;
      if (rank == 0) atomicCAS(p.status, 0, EBD_ERR_INVALID_ARG);
    }
    sm.r0 = r0;
    sm.n_rows = sm.bad_seq ? 0 : n;
    sm.meta_b = p.blk_meta[2 * seq];
    sm.meta_s = p.blk_meta[2 * seq + 1];
    sm.wait_fail = 0;
  }
  // every CTA of the cluster must be running before any distributed
  // shared-memory access; this also orders the block-level setup above
  cluster.sync();
  const int r0 = sm.r0, nr = sm.n_rows;

  for (int j = tid; j < nr; j += blockDim.x) {
    sm.f_mask[j] = p.mask[r0 + j];
    sm.f_ib[j] = p.in_block[r0 + j];
    sm.f_tok[j] = p.tokens[r0 + j];
    sm.f_pos[j] = p.row_pos[r0 + j];
    sm.f_acc[j] = 0;
    sm.f_O[j] = __int_as_float(0x7fc00000);
    sm.f_p[j] = __int_as_float(0x7fc00000);
  }

  // ---------------------------------------------------------------- 1. statistics
  if (p.features_in) {
    for (int j = tid; j < nr; j += blockDim.x) {
      const float c = p.conf[r0 + j], e = p.ent_norm[r0 + j], g = p.gap[r0 + j];
      const int a = p.argmax[r0 + j];
      sm.f_conf[j] = c;
      sm.f_ent[j] = e;
      sm.f_gap[j] = g;
      sm.f_arg[j] = a;
      sm.f_bad[j] = !(isfinite(c) && isfinite(e) && isfinite(g)) || a < 0 || a >= p.V;
    }
  } else {
    // row j is merged by warp (j / 8) of rank (j % 8) and broadcast
    for (int j = warp * kDecideCluster + rank; j < nr; j += kDecideCluster * (blockDim.x >> 5)) {
      const size_t base = static_cast<size_t>(r0 + j) * p.grid_lm;
      float m = -INFINITY, s = 0.f, t = 0.f, l2 = -INFINITY;
      int idx = INT_MAX;
      for (int g = lane; g < p.grid_lm; g += 32) {
        const float4 f = p.part_f[base + g];
        merge_state(m, s, t, l2, idx, f.x, f.y, f.z, f.w, p.part_i[base + g]);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float bm = __shfl_xor_sync(0xffffffffu, m, off);
        const float bs = __shfl_xor_sync(0xffffffffu, s, off);
        const float bt = __shfl_xor_sync(0xffffffffu, t, off);
        const float bl = __shfl_xor_sync(0xffffffffu, l2, off);
        const int bi = __shfl_xor_sync(0xffffffffu, idx, off);
        merge_state(m, s, t, l2, idx, bm, bs, bt, bl, bi);
      }
      const float conf = 1.0f / s;
      const float ent = logf(s) - t / s;
      const float entn = ent * p.inv_log_v;
      const float gap = (1.0f - expf(l2 - m)) / s;
      const bool bad = !(isfinite(m) && isfinite(s) && isfinite(t) && s >= 1.0f) || idx < 0 ||
                       idx >= p.V;
      if (lane == 0) {
        const int r = r0 + j;
        if (p.conf) p.conf[r] = conf;
        if (p.entropy) p.entropy[r] = ent;
        if (p.ent_norm) p.ent_norm[r] = entn;
        if (p.gap) p.gap[r] = gap;
        if (p.argmax) p.argmax[r] = bad ? -1 : idx;
        if (bad) atomicCAS(p.status, 0, EBD_ERR_NONFINITE);
      }
      if (lane < kDecideCluster) {
        Smem* dst = cluster.map_shared_rank(&sm, lane);
        dst->f_conf[j] = conf;
        dst->f_ent[j] = entn;
        dst->f_gap[j] = gap;
        dst->f_arg[j] = bad ? -1 : idx;
        dst->f_bad[j] = bad ? 1 : 0;
      }
    }
  }
  // the weight copy must have landed before any use (and before exit)
  {
    const bool ok = mbar_wait(&sm.bar, 0, 1000ull * 1000 * 1000, nullptr);
    if (!ok && tid == 0) {
      sm.wait_fail = 1;
      atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
    }
  }
  cluster.sync();

  // ---------------------------------------------------------------- 2. masked set
  if (tid == 0) {
    int nM = 0;
    for (int j = 0; j < nr; ++j)
      if (sm.f_mask[j]) sm.Mrows[nM++] = j;
    sm.nM = nM;
    sm.run_lbs = (sm.meta_s == 0 && nM > p.l_min) ? 1 : 0;
  }
  __syncthreads();
  const int nM = sm.nM;

  // ---------------------------------------------------------------- 3. LBS router
  if (sm.run_lbs) {
    const int n = nM;
    float* Z = P + P_Z;
    float* X = P + P_X;
    float* KV = P + P_KV;
    float* Q = P + P_Q;
    float* S = P + P_S;
    const float* Vv = sm.v;
    // 3a. entropy branch F_ent and token branch, every rank for all rows
    for (int it = tid; it < n * 64; it += blockDim.x) {
      const int j = it >> 6, o = it & 63;
      const int row = sm.Mrows[j];
      KV[j * LDKV + o] = gelu(fmaf(Vv[V_ENT1W + o], sm.f_ent[row], Vv[V_ENT1B + o]));
      const int tok = sm.f_arg[row];
      const float tv =
          (tok >= 0 && tok < p.V) ? p.w.tok_table[static_cast<size_t>(tok) * 64 + o] : 0.f;
      X[j * LDZ + 64 + o] = tv + Vv[V_TOKB + o];
    }
    __syncthreads();
    gemm_rows(KV, LDKV, n, 64, sm.w + W_ENT2, 64, 64, Vv + V_ENT2B,
              [&](int j, int o, float v) { X[j * LDZ + o] = v; });
    __syncthreads();
    layer_norm_rows(X, LDZ, X, LDZ, n, 64, Vv + V_ENTLNG, Vv + V_ENTLNB);
    __syncthreads();
    // 3b. fusion W_combine [e; t] + E_pos[rank of the row]: this CTA's 16 outputs
    {
      const int o0 = kCombSlice * rank;
      gemm_rows(X, LDZ, n, 128, sm.w + W_COMB, kCombSlice, kCombSlice, Vv + V_COMBB,
                [&](int j, int o, float v) {
                  const float val = v + __bfloat162float(sm.w[W_POS + j * kCombSlice + o]);
                  for (int rr = 0; rr < kDecideCluster; ++rr)
                    cluster.map_shared_rank(Z, rr)[j * LDZ + o0 + o] = val;
                });
    }
    cluster.sync();
    // 3c. two post-norm encoder layers
    const int hd = rank >> 1, half = rank & 1;
    const int nh = (n + 1) >> 1;
    const int qa = half == 0 ? 0 : nh, qb = half == 0 ? nh : n;
    for (int l = 0; l < 2; ++l) {
      const __nv_bfloat16* Wl = sm.w + W_LAYER0 + l * W_LAYER_STRIDE;
      const float* Vl = Vv + V_LAYER0 + l * V_LAYER_STRIDE;
      // QKV: this CTA's 48 features for every row, scattered to the CTAs
      // that attend with them (head h lives in ranks 2h and 2h+1)
      gemm_rows(Z, LDZ, n, 128, Wl + WL_QKV, kQkvSlice, kQkvSlice, Vl + VL_QKVB,
                [&](int j, int o, float v) {
                  const int f = kQkvSlice * rank + o;
                  const int part = f >> 7, h = (f >> 5) & 3, dd = f & 31;
                  if (part == 0) {
                    const int dst = 2 * h + (j >= nh ? 1 : 0);
                    const int jj = j >= nh ? j - nh : j;
                    cluster.map_shared_rank(P, dst)[P_Q + jj * LDQ + dd] = v;
                  } else {
                    const int col = (part == 1 ? 0 : 32) + dd;
                    cluster.map_shared_rank(P, 2 * h)[P_KV + j * LDKV + col] = v;
                    cluster.map_shared_rank(P, 2 * h + 1)[P_KV + j * LDKV + col] = v;
                  }
                });
      cluster.sync();
      attend(Q, LDQ, KV, KV + 32, LDKV, qb - qa, n, 32, S, [&](int i, int d, float v) {
        for (int rr = 0; rr < kDecideCluster; ++rr)
          cluster.map_shared_rank(X, rr)[(qa + i) * LDZ + 32 * hd + d] = v;
      });
      cluster.sync();
      {  // output projection + residual, 16 outputs, written in place into z
        const int o0 = kOutSlice * rank;
        gemm_rows(X, LDZ, n, 128, Wl + WL_OUT, kOutSlice, kOutSlice, Vl + VL_OUTB,
                  [&](int j, int o, float v) {
                    const float val = v + Z[j * LDZ + o0 + o];
                    for (int rr = 0; rr < kDecideCluster; ++rr)
                      cluster.map_shared_rank(Z, rr)[j * LDZ + o0 + o] = val;
                  });
      }
      cluster.sync();
      layer_norm_rows(Z, LDZ, Z, LDZ, n, 128, Vl + VL_LN1G, Vl + VL_LN1B);
      __syncthreads();
      // FFN: hidden units [32r, 32r+32) locally, then the partial second
      // linear of those units sent to the owners of each 16-output slice
      float* Hh = KV;  // [n][36]
      gemm_rows(Z, LDZ, n, 128, Wl + WL_FF1, kFf1Slice, kFf1Slice, Vl + VL_FF1B,
                [&](int j, int o, float v) { Hh[j * LDQ + o] = gelu(v); });
      __syncthreads();
      gemm_rows(Hh, LDQ, n, kFf1Slice, Wl + WL_FF2, 128, 128, nullptr,
                [&](int j, int o, float v) {
                  const int owner = o >> 4;
                  cluster.map_shared_rank(X, owner)[(rank * W + j) * 16 + (o & 15)] = v;
                });
      cluster.sync();
      {  // owner: sum the 8 partials + bias + residual, broadcast its slice
        const int o0 = kOutSlice * rank;
        for (int it = tid; it < n * 16; it += blockDim.x) {
          const int j = it >> 4, oo = it & 15;
          float a = Vl[VL_FF2B + oo] + Z[j * LDZ + o0 + oo];
#pragma unroll
          for (int src = 0; src < kDecideCluster; ++src) a += X[(src * W + j) * 16 + oo];
          for (int rr = 0; rr < kDecideCluster; ++rr)
            cluster.map_shared_rank(Z, rr)[j * LDZ + o0 + oo] = a;
        }
      }
      cluster.sync();
      layer_norm_rows(Z, LDZ, Z, LDZ, n, 128, Vl + VL_LN2G, Vl + VL_LN2B);
      __syncthreads();
    }
    // 3d. head Linear(128 -> 1), needed by rank 0
    if (rank == 0) {
      for (int j = warp; j < n; j += (blockDim.x >> 5)) {
        float a = 0.f;
        for (int c = 0; c < 4; ++c) a += Z[j * LDZ + lane + 32 * c] * Vv[V_HEADW + lane + 32 * c];
        a = warp_sum(a) + Vv[V_HEADB];
        if (lane == 0) sm.f_O[sm.Mrows[j]] = a;
      }
    }
    __syncthreads();
  }
  if (rank != 0) return;  // no distributed shared-memory access after this point

  // ---------------------------------------------------------------- 4. block selection
  if (tid == 0) {
    if (sm.meta_s == 0) {
      for (int j = 0; j < nr; ++j) sm.f_ib[j] = 0;
      int nB = 0;
      if (nM <= p.l_min) {
        for (int k = 0; k < nM; ++k) sm.Brows[nB++] = sm.Mrows[k];
      } else {
        int last = 0;
        for (int k = 0; k < nM; ++k) {
          const int j = sm.Mrows[k];
          const bool cand = sm.f_O[j] > 0.f && sm.f_arg[j] != p.eos_id && !sm.f_bad[j];
          if (!cand) continue;
          if (nB > 0 && sm.f_pos[j] - last > p.g_max) break;  // MaxGapFilter
          sm.Brows[nB++] = j;
          last = sm.f_pos[j];
        }
        if (nB < p.l_min) {  // min-tokens fallback
          nB = 0;
          const int take = nM < p.l_b ? nM : p.l_b;
          for (int k = 0; k < take; ++k) sm.Brows[nB++] = sm.Mrows[k];
        }
      }
      if (nB > 0) {
        for (int k = 0; k < nB; ++k) sm.f_ib[sm.Brows[k]] = 1;
        sm.meta_b = sm.f_pos[sm.Brows[0]];
        sm.meta_s = nB;
      }
    }
    int nBM = 0;
    for (int j = 0; j < nr; ++j)
      if (sm.f_ib[j] && sm.f_mask[j] && !sm.f_bad[j]) sm.BMrows[nBM++] = j;
    sm.nBM = nBM;
  }
  __syncthreads();

  // ---------------------------------------------------------------- 5. LPS + accept + commit
  const int nBM = sm.nBM;
  if (nBM > 0) {
    if (p.lps_enabled) lps_forward(sm, nBM);
    if (tid == 0) {
      int nacc = 0;
      for (int i = 0; i < nBM; ++i) {
        const int j = sm.BMrows[i];
        const bool a = sm.f_conf[j] >= p.tau || (p.lps_enabled && sm.f_p[j] > p.tau_psi);
        if (a) {
          sm.f_acc[j] = 1;
          ++nacc;
        }
      }
      if (nacc == 0) {  // anti-stall: highest confidence, lowest position on ties
        int best = sm.BMrows[0];
        for (int i = 1; i < nBM; ++i) {
          const int j = sm.BMrows[i];
          if (sm.f_conf[j] > sm.f_conf[best]) best = j;
        }
        sm.f_acc[best] = 1;
      }
      bool open = false;
      for (int j = 0; j < nr; ++j) {
        if (sm.f_acc[j]) {
          sm.f_tok[j] = sm.f_arg[j];
          sm.f_mask[j] = 0;
        }
        if (sm.f_ib[j] && sm.f_mask[j]) open = true;
      }
      if (sm.meta_s > 0 && !open) {
        for (int j = 0; j < nr; ++j) sm.f_ib[j] = 0;
        sm.meta_b = 0;
        sm.meta_s = 0;
      }
    }
  } else if (tid == 0 && sm.meta_s > 0) {
    bool open = false;
    for (int j = 0; j < nr; ++j)
      if (sm.f_ib[j] && sm.f_mask[j]) open = true;
    if (!open) {
      for (int j = 0; j < nr; ++j) sm.f_ib[j] = 0;
      sm.meta_b = 0;
      sm.meta_s = 0;
    }
  }
  __syncthreads();

  // ---------------------------------------------------------------- 6. write back
  for (int j = tid; j < nr; j += blockDim.x) {
    const int r = r0 + j;
    p.tokens[r] = sm.f_tok[j];
    p.mask[r] = sm.f_mask[j];
    p.in_block[r] = sm.f_ib[j];
    if (p.accepted) p.accepted[r] = sm.f_acc[j];
    if (p.lbs_logit) p.lbs_logit[r] = sm.f_O[j];
    if (p.lps_prob) p.lps_prob[r] = sm.f_p[j];
  }
  if (tid == 0 && !sm.bad_seq) {
    p.blk_meta[2 * seq] = sm.meta_b;
    p.blk_meta[2 * seq + 1] = sm.meta_s;
  }
}

// ----------------------------------------------------------------- token-branch fold
// table[v][j] = sum_k W_tok[j][k] W_e[v][k]  (fp32 accumulation)
__global__ void __launch_bounds__(256) fold_tok_kernel(const __nv_bfloat16* __restrict__ w_tok,
                                                        const __nv_bfloat16* __restrict__ w_emb,
                                                        float* __restrict__ table, int V,
                                                        int d_base) {
  __shared__ float sE[64][33];
  __shared__ float sW[64][33];
  const int v0 = blockIdx.x * 64;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;  // 16 x 16 threads, 4x4 outputs
  float acc[4][4] = {};
  for (int k0 = 0; k0 < d_base; k0 += 32) {
    for (int it = threadIdx.x; it < 64 * 32; it += 256) {
      const int r = it >> 5, c = it & 31;
      const int k = k0 + c;
      const int v = v0 + r;
      sE[r][c] = (v < V && k < d_base) ? __bfloat162float(w_emb[static_cast<size_t>(v) * d_base + k]) : 0.f;
      sW[r][c] = (k < d_base) ? __bfloat162float(w_tok[static_cast<size_t>(r) * d_base + k]) : 0.f;
    }
    __syncthreads();
    for (int c = 0; c < 32; ++c) {
      float e[4], ww[4];
      for (int i = 0; i < 4; ++i) e[i] = sE[ty * 4 + i][c];
      for (int i = 0; i < 4; ++i) ww[i] = sW[tx * 4 + i][c];
      for (int i = 0; i < 4; ++i)
        for (int jj = 0; jj < 4; ++jj) acc[i][jj] = fmaf(e[i], ww[jj], acc[i][jj]);
    }
    __syncthreads();
  }
  for (int i = 0; i < 4; ++i) {
    const int v = v0 + ty * 4 + i;
    if (v >= V) continue;
    for (int jj = 0; jj < 4; ++jj) table[static_cast<size_t>(v) * 64 + tx * 4 + jj] = acc[i][jj];
  }
}

// Merge of the LM-head partial states into the statistics, one warp per row
// (the statistics-only entry point).
__global__ void __launch_bounds__(256) merge_stats_kernel(const float4* __restrict__ part_f,
                                                          const int* __restrict__ part_i, int rows,
                                                          int grid, int V, float inv_log_v,
                                                          float* conf, float* entropy,
                                                          float* ent_norm, float* gap, int* argmax,
                                                          int* status) {
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (r >= rows) return;
  const size_t base = static_cast<size_t>(r) * grid;
  float m = -INFINITY, s = 0.f, t = 0.f, l2 = -INFINITY;
  int idx = INT_MAX;
  for (int g = lane; g < grid; g += 32) {
    const float4 f = part_f[base + g];
    merge_state(m, s, t, l2, idx, f.x, f.y, f.z, f.w, part_i[base + g]);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float bm = __shfl_xor_sync(0xffffffffu, m, off);
    const float bs = __shfl_xor_sync(0xffffffffu, s, off);
    const float bt = __shfl_xor_sync(0xffffffffu, t, off);
    const float bl = __shfl_xor_sync(0xffffffffu, l2, off);
    const int bi = __shfl_xor_sync(0xffffffffu, idx, off);
    merge_state(m, s, t, l2, idx, bm, bs, bt, bl, bi);
  }
  if (lane != 0) return;
  const float ent = logf(s) - t / s;
  const bool bad = !(isfinite(m) && isfinite(s) && isfinite(t) && s >= 1.0f) || idx < 0 || idx >= V;
  if (conf) conf[r] = 1.0f / s;
  if (entropy) entropy[r] = ent;
  if (ent_norm) ent_norm[r] = ent * inv_log_v;
  if (gap) gap[r] = (1.0f - expf(l2 - m)) / s;
  if (argmax) argmax[r] = bad ? -1 : idx;
  if (bad) atomicCAS(status, 0, EBD_ERR_NONFINITE);
}

cudaError_t launch_merge_stats(const float4* part_f, const int* part_i, int rows, int grid, int V,
                               float inv_log_v, float* conf, float* entropy, float* ent_norm,
                               float* gap, int* argmax, int* status, cudaStream_t st) {
  merge_stats_kernel<<<(rows + 7) / 8, 256, 0, st>>>(part_f, part_i, rows, grid, V, inv_log_v, conf,
                                                    entropy, ent_norm, gap, argmax, status);
  return cudaGetLastError();
}

cudaError_t decide_configure() {
  return cudaFuncSetAttribute(decide_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(sizeof(Smem) + 16));
}

cudaError_t launch_decide(const DecideParams& p, cudaStream_t st) {
  if (p.B <= 0) return cudaSuccess;
  decide_kernel<<<p.B * kDecideCluster, kDecideThreads, sizeof(Smem) + 16, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_fold_tok(const __nv_bfloat16* w_tok, const __nv_bfloat16* w_emb, float* table,
                            int V, int d_base, cudaStream_t st) {
  fold_tok_kernel<<<(V + 63) / 64, 256, 0, st>>>(w_tok, w_emb, table, V, d_base);
  return cudaGetLastError();
}

}  // namespace ebd
