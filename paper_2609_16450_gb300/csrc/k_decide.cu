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
// query half); every CTA keeps a full copy of the residual stream and the
// slices are exchanged through distributed shared memory.  The LPS router
// and the decision run in rank 0.
//
// Matrix products run on the tensor cores (mma.sync m16n8k16, bf16 weights,
// fp32 accumulation).  Every activation that feeds a product is stored once,
// by the phase that produces it, as a bf16 high part and a bf16 remainder
// (x = hi + lo to ~16 mantissa bits), so that a product loads its A fragments
// with ldmatrix and runs two MMAs per k-step.  The kernel is short and
// latency-bound: phases are kept few and their per-warp chains short.
#include <cooperative_groups.h>

#include <climits>

#include "decide_common.cuh"

namespace cg = cooperative_groups;

namespace ebd {

namespace {

// activation pool (floats), LBS phase
constexpr int P_Z = 0;                       // [64][132] fp32 residual stream z
constexpr int P_ZH = P_Z + W * LDZ;          // [64][136] bf16 x2: z as GEMM input (hi, lo)
constexpr int P_XH = P_ZH + W * LDH;         // [64][136] bf16 x2: [e;t] | concat ; fp32 FFN inbox [8][64][16]
constexpr int P_KV = P_XH + W * LDH;         // [64][68]  fp32 k,v of this CTA's head | bf16 x2 FFN hidden / F_ent
constexpr int P_Q = P_KV + W * LDKV;         // [32][36]  fp32 queries of this CTA's half
constexpr int P_S = P_Q + 32 * LDQ;          // [32][68]  fp32 attention scores
constexpr int POOL = P_S + 32 * LDS;
static_assert(8 * W * 16 <= W * LDH, "FFN partial inbox");
static_assert(W * 72 <= POOL - P_KV, "F_ent hidden hi/lo (spans k/v, q and scores)");
static_assert(W * LDZ <= W * LDH, "ent2 output scratch in the z hi/lo region");
static_assert(L_PROB + W <= POOL, "LPS pool layout");

struct __align__(16) Smem {
  __nv_bfloat16 w[LBS_W_ELEMS];  // this rank's LBS weight slices; later the LPS weights
  float v[V_ELEMS];              // vectors
  float pool[POOL];
  float f_conf[W], f_ent[W], f_gap[W], f_O[W], f_p[W];
  int f_arg[W], f_pos[W], f_tok[W], Mrows[W], Brows[W], BMrows[W];
  uint8_t f_mask[W], f_ib[W], f_acc[W], f_bad[W];
  int nM, nBM, meta_b, meta_s, n_rows, r0, run_lbs, bad_seq, lps_loaded;
  uint64_t bar;   // vectors (+ LBS weights)
  uint64_t bar2;  // LPS weights
};
static_assert(sizeof(Smem) + 16 <= 232448, "dynamic shared memory of one CTA");

// ------------------------------------------------------------------ LBS attention
// This CTA's query rows [qa, qa + nq) of head hd (width 32) over the n rows'
// keys/values: softmax(q k^T / sqrt(32)) v on the tensor cores.  q, k, v and
// the probabilities are split into bf16 high and low parts (three products
// per pair).  The work is spread over the warps: a warp takes one 16-query
// tile, one block of 16 keys and (when tiles x blocks leave warps idle) a
// group of the 8-column output tiles, and leaves its block's row max m, sum l
// and unnormalised output o in shared memory (the z hi/lo region, free
// between the QKV product and the next LayerNorm).  The whole CTA then
// combines the blocks, out = sum_b e^(m_b - M) o_b / sum_b e^(m_b - M) l_b,
// and writes the result as hi/lo, 16 bytes per store, into every rank's
// concat buffer.
constexpr int kAttLdp = 40;  // row stride of a partial output tile (floats)

__device__ __forceinline__ void lbs_attention(cg::cluster_group& cluster, float* P, int nq, int n,
                                              int qa, int hd) {
  const float* Q = P + P_Q;
  const float* KV = P + P_KV;
  float* part_o = P + P_ZH;                    // [unit][16][kAttLdp]
  float* part_ml = part_o + 8 * 16 * kAttLdp;  // [unit][16][2]
  static_assert(8 * 16 * (kAttLdp + 2) <= W * LDH, "attention partials fit the z hi/lo region");
  __nv_bfloat16* X = reinterpret_cast<__nv_bfloat16*>(P + P_XH);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const float scale = 0.17677669529663687f;  // 1/sqrt(32)
  const int mtq = (nq + 15) >> 4, nkb = (n + 15) >> 4;
  const int units = mtq * nkb;  // <= 2 x 4
  const int nsplit = units <= 2 ? 4 : (units <= 4 ? 2 : 1);
  if (warp < units * nsplit) {
    const int u = warp / nsplit, part = warp % nsplit;
    const int qt = u / nkb, kb = u % nkb;
    const int nt0 = part * (4 / nsplit), nt1 = nt0 + 4 / nsplit;
    const int r_lo = qt * 16 + g, r_hi = r_lo + 8;
    uint32_t qh[2][4], ql[2][4];
#pragma unroll
    for (int ks = 0; ks < 2; ++ks) {
      const float2 z = make_float2(0.f, 0.f);
      const float* ql0 = Q + r_lo * LDQ + 16 * ks + 2 * t;
      const float* qh0 = Q + r_hi * LDQ + 16 * ks + 2 * t;
      const float2 a0 = r_lo < nq ? *reinterpret_cast<const float2*>(ql0) : z;
      const float2 a1 = r_hi < nq ? *reinterpret_cast<const float2*>(qh0) : z;
      const float2 a2 = r_lo < nq ? *reinterpret_cast<const float2*>(ql0 + 8) : z;
      const float2 a3 = r_hi < nq ? *reinterpret_cast<const float2*>(qh0 + 8) : z;
      split_bf16x2(a0.x, a0.y, qh[ks][0], ql[ks][0]);
      split_bf16x2(a1.x, a1.y, qh[ks][1], ql[ks][1]);
      split_bf16x2(a2.x, a2.y, qh[ks][2], ql[ks][2]);
      split_bf16x2(a3.x, a3.y, qh[ks][3], ql[ks][3]);
    }
    const int k0 = 16 * kb;
    float s[2][4];
#pragma unroll
    for (int hb = 0; hb < 2; ++hb) {
      const int key = k0 + 8 * hb + g;
      float a[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int ks = 0; ks < 2; ++ks) {
        const float2 z = make_float2(0.f, 0.f);
        const float* kp = KV + key * LDKV + 16 * ks + 2 * t;
        const float2 k0v = key < n ? *reinterpret_cast<const float2*>(kp) : z;
        const float2 k1v = key < n ? *reinterpret_cast<const float2*>(kp + 8) : z;
        uint32_t bh0, bl0, bh1, bl1;
        split_bf16x2(k0v.x, k0v.y, bh0, bl0);
        split_bf16x2(k1v.x, k1v.y, bh1, bl1);
        mma_bf16(a, qh[ks], bh0, bh1);
        mma_bf16(a, qh[ks], bl0, bl1);
        mma_bf16(a, ql[ks], bh0, bh1);
      }
      const int c = k0 + 8 * hb + 2 * t;
      s[hb][0] = c < n ? a[0] * scale : -INFINITY;
      s[hb][1] = c + 1 < n ? a[1] * scale : -INFINITY;
      s[hb][2] = c < n ? a[2] * scale : -INFINITY;
      s[hb][3] = c + 1 < n ? a[3] * scale : -INFINITY;
    }
    float m0 = fmaxf(fmaxf(s[0][0], s[0][1]), fmaxf(s[1][0], s[1][1]));
    float m1 = fmaxf(fmaxf(s[0][2], s[0][3]), fmaxf(s[1][2], s[1][3]));
    m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, 1));
    m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, 2));
    m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, 1));
    m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, 2));  // finite: key k0 is valid
#pragma unroll
    for (int hb = 0; hb < 2; ++hb) {
      s[hb][0] = expf(s[hb][0] - m0);
      s[hb][1] = expf(s[hb][1] - m0);
      s[hb][2] = expf(s[hb][2] - m1);
      s[hb][3] = expf(s[hb][3] - m1);
    }
    uint32_t ph[4], pl[4];
    split_bf16x2(s[0][0], s[0][1], ph[0], pl[0]);
    split_bf16x2(s[0][2], s[0][3], ph[1], pl[1]);
    split_bf16x2(s[1][0], s[1][1], ph[2], pl[2]);
    split_bf16x2(s[1][2], s[1][3], ph[3], pl[3]);
    float* po = part_o + u * 16 * kAttLdp;
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
      if (nt < nt0 || nt >= nt1) continue;
      float o[4] = {0.f, 0.f, 0.f, 0.f};
      float v[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = k0 + (e >> 1) * 8 + 2 * t + (e & 1);
        v[e] = key < n ? KV[key * LDKV + 32 + 8 * nt + g] : 0.f;
      }
      uint32_t v0h, v0l, v1h, v1l;
      split_bf16x2(v[0], v[1], v0h, v0l);
      split_bf16x2(v[2], v[3], v1h, v1l);
      mma_bf16(o, ph, v0h, v1h);
      mma_bf16(o, ph, v0l, v1l);
      mma_bf16(o, pl, v0h, v1h);
      *reinterpret_cast<float2*>(po + g * kAttLdp + 8 * nt + 2 * t) = make_float2(o[0], o[1]);
      *reinterpret_cast<float2*>(po + (g + 8) * kAttLdp + 8 * nt + 2 * t) = make_float2(o[2], o[3]);
    }
    if (part == 0) {
      float l0 = (s[0][0] + s[0][1]) + (s[1][0] + s[1][1]);
      float l1 = (s[0][2] + s[0][3]) + (s[1][2] + s[1][3]);
      l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
      l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
      l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
      l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
      if (t == 0) {
        float* pm = part_ml + u * 32;
        *reinterpret_cast<float2*>(pm + 2 * g) = make_float2(m0, l0);
        *reinterpret_cast<float2*>(pm + 2 * (g + 8)) = make_float2(m1, l1);
      }
    }
  }
  __syncthreads();
  // combine: one thread per (query row, 8 output columns), both planes to
  // every rank (this one included)
#pragma unroll 1
  for (int it = threadIdx.x; it < nq * 4; it += blockDim.x) {
    const int r = it >> 2, c8 = it & 3, qt = r >> 4, rr = r & 15;
    float M = -INFINITY;
#pragma unroll 1
    for (int kb = 0; kb < nkb; ++kb) M = fmaxf(M, part_ml[(qt * nkb + kb) * 32 + 2 * rr]);
    float L = 0.f, acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
    for (int kb = 0; kb < nkb; ++kb) {
      const int u = qt * nkb + kb;
      const float2 ml = *reinterpret_cast<const float2*>(part_ml + u * 32 + 2 * rr);
      const float e = expf(ml.x - M);
      L = fmaf(e, ml.y, L);
      const float4* src = reinterpret_cast<const float4*>(part_o + (u * 16 + rr) * kAttLdp + 8 * c8);
      const float4 x0 = src[0], x1 = src[1];
      acc[0] = fmaf(e, x0.x, acc[0]);
      acc[1] = fmaf(e, x0.y, acc[1]);
      acc[2] = fmaf(e, x0.z, acc[2]);
      acc[3] = fmaf(e, x0.w, acc[3]);
      acc[4] = fmaf(e, x1.x, acc[4]);
      acc[5] = fmaf(e, x1.y, acc[5]);
      acc[6] = fmaf(e, x1.z, acc[6]);
      acc[7] = fmaf(e, x1.w, acc[7]);
    }
    const float iL = 1.0f / L;
    uint4 hi, lo;
    split_bf16x2(acc[0] * iL, acc[1] * iL, hi.x, lo.x);
    split_bf16x2(acc[2] * iL, acc[3] * iL, hi.y, lo.y);
    split_bf16x2(acc[4] * iL, acc[5] * iL, hi.z, lo.z);
    split_bf16x2(acc[6] * iL, acc[7] * iL, hi.w, lo.w);
    const int off = (qa + r) * LDH + 32 * hd + 8 * c8;
#pragma unroll 1
    for (int rk = 0; rk < kDecideCluster; ++rk) {
      __nv_bfloat16* dst = cluster.map_shared_rank(X, rk);
      *reinterpret_cast<uint4*>(dst + off) = hi;
      *reinterpret_cast<uint4*>(dst + W * LDH + off) = lo;
    }
  }
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
  // a kernel launched after this one as a programmatic dependent (the window
  // attention, which shares no data with the decision) may start on the SMs
  // this grid leaves free once every CTA of it is resident
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (tid == 0) {
    // weights and vectors of this rank: bulk copies issued first, so they
    // land while the statistics are merged.  With no active block the LBS
    // weights are needed (every rank); otherwise only rank 0 needs the LPS
    // weights, which then go straight into the weight region.
    mbar_init(&sm.bar, 1);
    mbar_init(&sm.bar2, 1);
    fence_mbar_init();
    sm.meta_b = p.blk_meta[2 * seq];
    sm.meta_s = p.blk_meta[2 * seq + 1];
    const bool lbs_possible = p.mode == EBD_DECODE_EB && sm.meta_s == 0;
    const uint32_t wb = LBS_W_ELEMS * 2u, vb = V_ELEMS * 4u;
    mbar_arrive_expect_tx(&sm.bar, vb + (lbs_possible ? wb : 0u));
    bulk_copy(sm.v, p.w.vec + static_cast<size_t>(rank) * V_ELEMS, vb, &sm.bar);
    if (lbs_possible)
      bulk_copy(sm.w, p.w.lbs_w + static_cast<size_t>(rank) * LBS_W_ELEMS, wb, &sm.bar);
    sm.lps_loaded = 0;
    if (!lbs_possible && rank == 0 && p.lps_enabled) {
      mbar_arrive_expect_tx(&sm.bar2, LPS_W_ELEMS * 2u);
      bulk_copy(sm.w, p.w.lps_w, LPS_W_ELEMS * 2u, &sm.bar2);
      sm.lps_loaded = 1;
    }
    const int r0 = p.cu_rows[seq], r1 = p.cu_rows[seq + 1];
    const int n = r1 - r0;
    sm.bad_seq = 0;
    if (p.cu_rows[p.B] != p.rows_expected || n < 0 || n > W || r0 < 0) {
      sm.bad_seq = 1;
      if (rank == 0) atomicCAS(p.status, 0, EBD_ERR_INVALID_ARG);
    }
    sm.r0 = r0;
    sm.n_rows = sm.bad_seq ? 0 : n;
  }
  // every CTA of the cluster must be running before any distributed
  // shared-memory access; this also orders the block-level setup above
  cluster.sync();
  const int r0 = sm.r0, nr = sm.n_rows;

#pragma unroll 1
  for (int j = tid; j < nr; j += blockDim.x) {
    sm.f_mask[j] = p.mask[r0 + j];
    sm.f_ib[j] = p.in_block[r0 + j];
    sm.f_tok[j] = p.tokens[r0 + j];
    sm.f_pos[j] = p.row_pos[r0 + j];
    sm.f_acc[j] = 0;
    sm.f_O[j] = __int_as_float(0x7fc00000);
    sm.f_p[j] = __int_as_float(0x7fc00000);
  }

  // Every step starts with this kernel's code out of every cache.  While the
  // LM head finishes, ranks 1..5 each run one stretch of the LPS router on a
  // stand-in block in their own shared memory (the pool, unused until the
  // statistics are merged; the results are discarded), so that the
  // instructions rank 0 runs there after the LBS come from L2.
  if (rank >= 1 && rank <= 5 && p.lps_enabled && p.mode == EBD_DECODE_EB) {
    const int from = rank == 1 ? 0 : rank == 2 ? 1 : rank == 3 ? 3 : rank == 4 ? 4 : 6;
    const int to = rank == 1 ? 0 : rank == 2 ? 2 : rank == 3 ? 3 : rank == 4 ? 5 : 7;
    lps_forward(P, 32, sm.w, sm.v + V_LPS, from, to);
  }

  // ---------------------------------------------------------------- 1. statistics
  // Launched as a programmatic dependent of the LM head, the kernel may start
  // while the LM head's last CTAs run: everything above (weights in flight,
  // decode state loaded) overlaps them; the partial states are read only
  // after the LM head's grid has completed and its writes are visible.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (p.features_in) {
#pragma unroll 1
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
#pragma unroll 1
    for (int j = warp * kDecideCluster + rank; j < nr; j += kDecideCluster * (blockDim.x >> 5)) {
      const size_t base = static_cast<size_t>(r0 + j) * p.grid_lm;
      float m = -INFINITY, s = 0.f, t = 0.f, l2 = -INFINITY;
      int idx = INT_MAX;
      float4 fv[8];
      int iv[8];
#pragma unroll
      for (int c = 0; c < 8; ++c) {  // independent loads first (partials per lane <= 8)
        const int g = lane + 32 * c;
        fv[c] = g < p.grid_lm ? p.part_f[base + g] : make_float4(-INFINITY, 0.f, 0.f, -INFINITY);
        iv[c] = g < p.grid_lm ? p.part_i[base + g] : INT_MAX;
      }
#pragma unroll
      for (int c = 0; c < 8; ++c)
        merge_state(m, s, t, l2, idx, fv[c].x, fv[c].y, fv[c].z, fv[c].w, iv[c]);
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
      if (lane == 0 && in_bounds(r0 + j, p.rows_expected, p.status)) {
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
  if (!mbar_wait(&sm.bar, 0, 1000ull * 1000 * 1000, nullptr) && tid == 0)
    atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
  cluster.sync();

  // ---------------------------------------------------------------- 2. masked set
  if (warp == 0) {
    int base = 0;
#pragma unroll 1
    for (int j0 = 0; j0 < nr; j0 += 32) {
      const int j = j0 + lane;
      const bool m = j < nr && sm.f_mask[j];
      const uint32_t bal = __ballot_sync(0xffffffffu, m);
      if (m) sm.Mrows[base + __popc(bal & ((1u << lane) - 1u))] = j;
      base += __popc(bal);
    }
    if (lane == 0) {
      sm.nM = base;
      sm.run_lbs = (p.mode == EBD_DECODE_EB && sm.meta_s == 0 && base > p.l_min) ? 1 : 0;
    }
  }
  __syncthreads();
  const int nM = sm.nM;

  // ---------------------------------------------------------------- 3. LBS router
  if (sm.run_lbs) {
    const int n = nM;
    float* Z = P + P_Z;
    const HL Zh = hl_at(P + P_ZH, LDH);
    const HL Xh = hl_at(P + P_XH, LDH);
    float* Xin = P + P_XH;  // fp32 FFN partial inbox [8][64][16] (aliases Xh)
    const HL Fh = hl_at(P + P_KV, 72);  // F_ent hidden (hi/lo)
    const HL Hh = hl_at(P + P_KV, 40);  // FFN hidden slice (hi/lo)
    float* KV = P + P_KV;
    float* Q = P + P_Q;
    const float* Vv = sm.v;
    // 3a. entropy branch F_ent and token branch, every rank for all rows.
    // The token branch's gathers from the folded table are issued first and
    // stored only after the entropy branch, which hides their latency.
    static_assert(kDecideThreads * 8 >= W * 32, "token-branch items per thread");
    float2 tv[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int it = tid + k * kDecideThreads;
      tv[k] = make_float2(0.f, 0.f);
      if (it < n * 32) {
        const int tok = sm.f_arg[sm.Mrows[it >> 5]];
        if (tok >= 0 && tok < p.V)
          tv[k] = __ldg(reinterpret_cast<const float2*>(p.w.tok_table + static_cast<size_t>(tok) * 64 +
                                                       2 * (it & 31)));
      }
    }
#pragma unroll 1
    for (int it = tid; it < n * 32; it += blockDim.x) {
      const int j = it >> 5, o = 2 * (it & 31);
      const float h = sm.f_ent[sm.Mrows[j]];
      hl_store2(Fh, j, o, gelu(fmaf(Vv[V_ENT1W + o], h, Vv[V_ENT1B + o])),
                gelu(fmaf(Vv[V_ENT1W + o + 1], h, Vv[V_ENT1B + o + 1])));
    }
    __syncthreads();
    // the ent2 output goes to the z hi/lo region: z itself receives the
    // other ranks' fusion outputs as soon as they get there
    float* E2 = P + P_ZH;
    gemm_hl<true>(Fh, n, 64, sm.w + W_ENT2, 64, 64, [&](int j, int o, float a, float b) {
      *reinterpret_cast<float2*>(E2 + j * LDZ + o) = make_float2(a + Vv[V_ENT2B + o], b + Vv[V_ENT2B + o + 1]);
    });
    __syncthreads();
    ln_rows<64, false>(E2, LDZ, nullptr, 0, Xh, n, Vv + V_ENTLNG, Vv + V_ENTLNB);
#pragma unroll
    for (int k = 0; k < 8; ++k) {  // the token branch into columns 64..127
      const int it = tid + k * kDecideThreads;
      if (it < n * 32) {
        const int o = 2 * (it & 31);
        hl_store2(Xh, it >> 5, 64 + o, tv[k].x + Vv[V_TOKB + o], tv[k].y + Vv[V_TOKB + o + 1]);
      }
    }
    __syncthreads();
    // 3b. fusion W_combine [e; t] + E_pos[rank of the row]: this CTA's 16 outputs
    {
      const int o0 = kCombSlice * rank;
      gemm_hl<true>(Xh, n, 128, sm.w + W_COMB, kCombSlice, kCombSlice, [&](int j, int o, float a, float b) {
        const float2 pe = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(sm.w + W_POS + j * kCombSlice + o));
        const float2 val = make_float2(a + Vv[V_COMBB + o] + pe.x, b + Vv[V_COMBB + o + 1] + pe.y);
#pragma unroll 1
        for (int r = 0; r < kDecideCluster; ++r)
          *reinterpret_cast<float2*>(cluster.map_shared_rank(Z, r) + j * LDZ + o0 + o) = val;
      });
    }
    cluster.sync();
    // z as the first QKV input (hi/lo), every rank for all rows
#pragma unroll 1
    for (int it = tid; it < n * 64; it += blockDim.x) {
      const int j = it >> 6, o = 2 * (it & 63);
      hl_store2(Zh, j, o, Z[j * LDZ + o], Z[j * LDZ + o + 1]);
    }
    __syncthreads();
    // 3c. two post-norm encoder layers
    const int hd = rank >> 1, half = rank & 1;
    const int nh = (n + 1) >> 1;
    const int qa = half == 0 ? 0 : nh, qb = half == 0 ? nh : n;
#pragma unroll 1
    for (int l = 0; l < 2; ++l) {
      const __nv_bfloat16* Wl = sm.w + W_LAYER0 + l * W_LAYER_STRIDE;
      const float* Vl = Vv + V_LAYER0 + l * V_LAYER_STRIDE;
      // QKV: this CTA's 48 features for every row, scattered to the CTAs
      // that attend with them (head h lives in ranks 2h and 2h+1)
      gemm_hl<true>(Zh, n, 128, Wl + WL_QKV, kQkvSlice, kQkvSlice, [&](int j, int o, float a, float b) {
        const int f = kQkvSlice * rank + o;  // even; f and f+1 share part and head
        const int part = f >> 7, h = (f >> 5) & 3, dd = f & 31;
        const float2 val = make_float2(a + Vl[VL_QKVB + o], b + Vl[VL_QKVB + o + 1]);
        if (part == 0) {
          const int dst = 2 * h + (j >= nh ? 1 : 0);
          const int jj = j >= nh ? j - nh : j;
          *reinterpret_cast<float2*>(cluster.map_shared_rank(Q, dst) + jj * LDQ + dd) = val;
        } else {
          const int col = (part == 1 ? 0 : 32) + dd;
          *reinterpret_cast<float2*>(cluster.map_shared_rank(KV, 2 * h) + j * LDKV + col) = val;
          *reinterpret_cast<float2*>(cluster.map_shared_rank(KV, 2 * h + 1) + j * LDKV + col) = val;
        }
      });
      cluster.sync();
      lbs_attention(cluster, P, qb - qa, n, qa, hd);
      cluster.sync();
      {  // output projection + residual, 16 outputs, written in place into z
        const int o0 = kOutSlice * rank;
        gemm_hl<true>(Xh, n, 128, Wl + WL_OUT, kOutSlice, kOutSlice, [&](int j, int o, float a, float b) {
          const float2 zz = *reinterpret_cast<const float2*>(Z + j * LDZ + o0 + o);
          const float2 val = make_float2(zz.x + (a + Vl[VL_OUTB + o]), zz.y + (b + Vl[VL_OUTB + o + 1]));
#pragma unroll 1
          for (int r = 0; r < kDecideCluster; ++r)
            *reinterpret_cast<float2*>(cluster.map_shared_rank(Z, r) + j * LDZ + o0 + o) = val;
        });
      }
      cluster.sync();
      ln_rows<128, true>(Z, LDZ, Z, LDZ, Zh, n, Vl + VL_LN1G, Vl + VL_LN1B);
      __syncthreads();
      // FFN: hidden units [32r, 32r+32) locally, then the partial second
      // linear of those units sent to the owners of each 16-output slice
      gemm_hl<true>(Zh, n, 128, Wl + WL_FF1, kFf1Slice, kFf1Slice, [&](int j, int o, float a, float b) {
        hl_store2(Hh, j, o, gelu(a + Vl[VL_FF1B + o]), gelu(b + Vl[VL_FF1B + o + 1]));
      });
      __syncthreads();
      gemm_hl<true>(Hh, n, kFf1Slice, Wl + WL_FF2, 128, 128, [&](int j, int o, float a, float b) {
        *reinterpret_cast<float2*>(cluster.map_shared_rank(Xin, o >> 4) + (rank * W + j) * 16 + (o & 15)) =
            make_float2(a, b);
      });
      cluster.sync();
      {  // owner: sum the 8 partials + bias + residual, broadcast its slice
        const int o0 = kOutSlice * rank;
#pragma unroll 1
        for (int it = tid; it < n * 8; it += blockDim.x) {
          const int j = it >> 3, oo = 2 * (it & 7);
          float2 a = *reinterpret_cast<const float2*>(Z + j * LDZ + o0 + oo);
          a.x += Vl[VL_FF2B + oo];
          a.y += Vl[VL_FF2B + oo + 1];
#pragma unroll
          for (int src = 0; src < kDecideCluster; ++src) {
            const float2 q = *reinterpret_cast<const float2*>(Xin + (src * W + j) * 16 + oo);
            a.x += q.x;
            a.y += q.y;
          }
#pragma unroll 1
          for (int rr = 0; rr < kDecideCluster; ++rr)
            *reinterpret_cast<float2*>(cluster.map_shared_rank(Z, rr) + j * LDZ + o0 + oo) = a;
        }
      }
      cluster.sync();
      ln_rows<128, true>(Z, LDZ, Z, LDZ, Zh, n, Vl + VL_LN2G, Vl + VL_LN2B);
      __syncthreads();
      if (l == 0 && rank == 0 && tid == 0 && p.lps_enabled) {
        // the first layer's weights (and everything before them) are dead:
        // fetch the LPS weights into that region behind the second layer
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        mbar_arrive_expect_tx(&sm.bar2, LPS_W_ELEMS * 2u);
        bulk_copy(sm.w, p.w.lps_w, LPS_W_ELEMS * 2u, &sm.bar2);
        sm.lps_loaded = 1;
      }
    }
    // 3d. head Linear(128 -> 1), needed by rank 0
    if (rank == 0) {
#pragma unroll 1
      for (int j = warp; j < n; j += (blockDim.x >> 5)) {
        float a = 0.f;
#pragma unroll
        for (int c = 0; c < 4; ++c) a += Z[j * LDZ + lane + 32 * c] * Vv[V_HEADW + lane + 32 * c];
        a = warp_sum(a) + Vv[V_HEADB];
        if (lane == 0) sm.f_O[sm.Mrows[j]] = a;
      }
    }
    __syncthreads();
  }
  // No distributed shared-memory access after this point.  Rank 0 makes the
  // decision.  Ranks 1..7 make none: each runs a part of the LPS router, or
  // the accept step, on a stand-in block of its own shared memory, skipping
  // the block selection and writing nothing to global memory.  Every step
  // starts with this kernel's code out of every cache; ahead of rank 0 and in
  // parallel, those runs bring the code rank 0 is about to execute into L2.
  const bool shadow = rank != 0;

  // ---------------------------------------------------------------- 4. block selection
  if (tid == 0 && !sm.lps_loaded && p.lps_enabled) {
    // no LBS ran: the weight region is free now
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    mbar_arrive_expect_tx(&sm.bar2, LPS_W_ELEMS * 2u);
    bulk_copy(sm.w, p.w.lps_w, LPS_W_ELEMS * 2u, &sm.bar2);
    sm.lps_loaded = 1;
  }
  if (warp == 0) {
    if (shadow) {
      // stand-in block: the first min(32, |M|) masked rows
      const int nB = nM < 32 ? nM : 32;
      for (int j = lane; j < nr; j += 32) sm.f_ib[j] = 0;
      __syncwarp();
      for (int k = lane; k < nB; k += 32) sm.f_ib[sm.Mrows[k]] = 1;
      if (lane == 0 && nB > 0) {
        sm.meta_b = sm.f_pos[sm.Mrows[0]];
        sm.meta_s = nB;
      }
      __syncwarp();
    } else if (p.mode != EBD_DECODE_EB) {
      // baselines: the window is the active fixed block; no block state
    } else if (sm.meta_s == 0) {
      for (int j = lane; j < nr; j += 32) sm.f_ib[j] = 0;
      __syncwarp();
      int nB = 0;
      if (nM <= p.l_min) {
        for (int k = lane; k < nM; k += 32) sm.Brows[k] = sm.Mrows[k];
        nB = nM;
      } else {
        // candidates (router O > 0, not EOS) compacted in ascending position
        int nC = 0;
        for (int k0 = 0; k0 < nM; k0 += 32) {
          const int k = k0 + lane;
          int j = -1;
          bool c = false;
          if (k < nM) {
            j = sm.Mrows[k];
            c = sm.f_O[j] > 0.f && sm.f_arg[j] != p.eos_id && !sm.f_bad[j];
          }
          const uint32_t bal = __ballot_sync(0xffffffffu, c);
          if (c) sm.Brows[nC + __popc(bal & ((1u << lane) - 1u))] = j;
          nC += __popc(bal);
        }
        __syncwarp();
        // MaxGapFilter: cut at the first candidate farther than g_max from its predecessor
        int cut = nC;
        for (int c0 = 1; c0 < nC; c0 += 32) {
          const int c = c0 + lane;
          const bool gap = c < nC && sm.f_pos[sm.Brows[c]] - sm.f_pos[sm.Brows[c - 1]] > p.g_max;
          const uint32_t bal = __ballot_sync(0xffffffffu, gap);
          if (bal) {
            cut = c0 + __ffs(bal) - 1;
            break;
          }
        }
        nB = cut;
        if (nB < p.l_min) {  // min-tokens fallback: first min(L_B, |M|) masked rows
          nB = nM < p.l_b ? nM : p.l_b;
          __syncwarp();
          for (int k = lane; k < nB; k += 32) sm.Brows[k] = sm.Mrows[k];
        }
      }
      __syncwarp();
      for (int k = lane; k < nB; k += 32) sm.f_ib[sm.Brows[k]] = 1;
      if (lane == 0 && nB > 0) {
        sm.meta_b = sm.f_pos[sm.Brows[0]];
        sm.meta_s = nB;
      }
      __syncwarp();
    }
    int base = 0;
    for (int j0 = 0; j0 < nr; j0 += 32) {
      const int j = j0 + lane;
      const bool inb = p.mode != EBD_DECODE_EB || sm.f_ib[j];
      const bool m = j < nr && inb && sm.f_mask[j] && !sm.f_bad[j];
      const uint32_t bal = __ballot_sync(0xffffffffu, m);
      if (m) sm.BMrows[base + __popc(bal & ((1u << lane) - 1u))] = j;
      base += __popc(bal);
    }
    if (lane == 0) sm.nBM = base;
  }
  __syncthreads();

  // ---------------------------------------------------------------- 5. LPS + accept + commit
  // the LPS weight copy must have landed before use and before exit
  if (sm.lps_loaded && !mbar_wait(&sm.bar2, 0, 1000ull * 1000 * 1000, nullptr))
    atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
  const int nBM = sm.nBM;
  // phase of the LPS router where a stand-in run starts (-1: accept only)
  const int lps_from = !shadow ? 0 : (rank <= 4 ? rank - 1 : (rank == 5 ? 4 : (rank == 6 ? 6 : -1)));
  if (nBM > 0 && p.lps_enabled && lps_from >= 0) {
    float* feats = P + L_FEAT;
    const float rho = static_cast<float>(nBM) / static_cast<float>(sm.meta_s);
#pragma unroll 1
    for (int i = tid; i < nBM; i += blockDim.x) {
      const int r = sm.BMrows[i];
      feats[i * 8 + 0] = sm.f_conf[r];
      feats[i * 8 + 1] = sm.f_ent[r];
      feats[i * 8 + 2] = sm.f_gap[r];
      feats[i * 8 + 3] = rho;
      feats[i * 8 + 4] = static_cast<float>(sm.f_pos[r] - sm.meta_b) / static_cast<float>(sm.meta_s);
    }
    __syncthreads();
    const float* prob = P + L_PROB;
    lps_forward(P, nBM, sm.w, sm.v + V_LPS, lps_from, 8);
#pragma unroll 1
    for (int i = tid; i < nBM; i += blockDim.x) sm.f_p[sm.BMrows[i]] = prob[i];
    __syncthreads();
  }
  if (warp == 0 && p.mode == EBD_DECODE_TOPM) {
    // Top-m (App. B, Eq. prelim-update): the rank of a row is the number of
    // rows ahead of it (higher kappa, or equal kappa and lower position)
    for (int i = lane; i < nBM; i += 32) {
      const int j = sm.BMrows[i];
      const float c = sm.f_conf[j];
      int rank = 0;
      for (int k = 0; k < nBM; ++k) {
        const int jk = sm.BMrows[k];
        const float ck = sm.f_conf[jk];
        rank += (ck > c || (ck == c && jk < j)) ? 1 : 0;
      }
      if (rank < p.top_m) sm.f_acc[j] = 1;
    }
    __syncwarp();
    for (int j = lane; j < nr; j += 32)
      if (sm.f_acc[j]) {
        sm.f_tok[j] = sm.f_arg[j];
        sm.f_mask[j] = 0;
      }
  } else if (warp == 0) {
    // union accept rule, anti-stall fallback, parallel commit, resolution
    bool any = false;
    for (int i0 = 0; i0 < nBM; i0 += 32) {
      const int i = i0 + lane;
      bool a = false;
      if (i < nBM) {
        const int j = sm.BMrows[i];
        a = sm.f_conf[j] >= p.tau || (p.lps_enabled && sm.f_p[j] > p.tau_psi);
        if (a) sm.f_acc[j] = 1;
      }
      any |= __ballot_sync(0xffffffffu, a) != 0;
    }
    if (!any && nBM > 0) {
      // highest confidence; the lowest position among equal confidences
      float best = -INFINITY;
      int bj = INT_MAX;
      for (int i = lane; i < nBM; i += 32) {
        const int j = sm.BMrows[i];
        const float c = sm.f_conf[j];
        if (c > best || (c == best && j < bj)) {
          best = c;
          bj = j;
        }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float ob = __shfl_xor_sync(0xffffffffu, best, off);
        const int oj = __shfl_xor_sync(0xffffffffu, bj, off);
        if (ob > best || (ob == best && oj < bj)) {
          best = ob;
          bj = oj;
        }
      }
      if (lane == 0) sm.f_acc[bj] = 1;
    }
    __syncwarp();
    bool open = false;
    for (int j0 = 0; j0 < nr; j0 += 32) {
      const int j = j0 + lane;
      if (j < nr) {
        if (sm.f_acc[j]) {
          sm.f_tok[j] = sm.f_arg[j];
          sm.f_mask[j] = 0;
        }
        open |= sm.f_ib[j] && sm.f_mask[j];
      }
    }
    open = __ballot_sync(0xffffffffu, open) != 0;
    if (p.mode == EBD_DECODE_EB && sm.meta_s > 0 && !open) {
      for (int j = lane; j < nr; j += 32) sm.f_ib[j] = 0;
      if (lane == 0) {
        sm.meta_b = 0;
        sm.meta_s = 0;
      }
    }
  }
  __syncthreads();

  // ---------------------------------------------------------------- 6. write back
  if (shadow) return;
  for (int j = tid; j < nr; j += blockDim.x) {
    const int r = r0 + j;
    if (!in_bounds(r, p.rows_expected, p.status)) continue;
    p.tokens_out[r] = sm.f_tok[j];
    p.mask_out[r] = sm.f_mask[j];
    p.in_block_out[r] = sm.f_ib[j];
    if (p.accepted) p.accepted[r] = sm.f_acc[j];
    if (p.lbs_logit) p.lbs_logit[r] = sm.f_O[j];
    if (p.lps_prob) p.lps_prob[r] = sm.f_p[j];
  }
  if (tid == 0 && !sm.bad_seq) {
    p.blk_meta_out[2 * seq] = sm.meta_b;
    p.blk_meta_out[2 * seq + 1] = sm.meta_s;
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
  // as a programmatic dependent of the LM head: its partial states are read
  // only after its grid completed; the grid-wide decision's chain follows
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
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
                               float* gap, int* argmax, int* status, cudaStream_t st, bool pdl) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>((rows + 7) / 8));
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, merge_stats_kernel, part_f, part_i, rows, grid, V, inv_log_v, conf,
                            entropy, ent_norm, gap, argmax, status);
}

// Vocabulary-parallel LM head (several GPUs, each holding a range of W's
// rows).  The softmax statistics of App. B (Eq. app-confidence), Sec. 5.1
// and Sec. 5.2 are functions of the whole vocabulary; each shard reduces its
// range to one online-softmax state per row (m, S, T, l2, x_hat), and the
// merge of states is associative, so the states of the shards, gathered on
// every GPU, merge into the statistics of the whole vocabulary.
//
// shard_state_kernel: one warp per row merges the row's `grid` LM-head
// partials into one state, stored as 8 words: m, S, T, l2, idx (int32 bits),
// and three zero words (32-byte rows).
__global__ void __launch_bounds__(256) shard_state_kernel(const float4* __restrict__ part_f,
                                                          const int* __restrict__ part_i, int rows,
                                                          int grid, float* __restrict__ state) {
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
  float4* o = reinterpret_cast<float4*>(state + static_cast<size_t>(r) * 8);
  o[0] = make_float4(m, s, t, l2);
  o[1] = make_float4(__int_as_float(idx), 0.f, 0.f, 0.f);
}

// merge_shards_kernel: one warp per row merges the row's state from each of
// `shards` shards (states[shard][row][8]) and writes the statistics as the
// merge of the single-GPU path does (kappa = 1/S, H = ln S - T/S,
// H~ = H / ln V with V the whole vocabulary, Delta = (1 - exp(l2 - m)) / S,
// x_hat = idx); a non-finite state records EBD_ERR_NONFINITE.
__global__ void __launch_bounds__(256) merge_shards_kernel(const float* __restrict__ states,
                                                           int shards, int rows, int V,
                                                           float inv_log_v, float* conf,
                                                           float* entropy, float* ent_norm,
                                                           float* gap, int* argmax, int* status) {
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (r >= rows) return;
  float m = -INFINITY, s = 0.f, t = 0.f, l2 = -INFINITY;
  int idx = INT_MAX;
  for (int g = lane; g < shards; g += 32) {
    const float4* q = reinterpret_cast<const float4*>(
        states + (static_cast<size_t>(g) * rows + r) * 8);
    const float4 f = q[0];
    const float4 i4 = q[1];
    merge_state(m, s, t, l2, idx, f.x, f.y, f.z, f.w, __float_as_int(i4.x));
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

cudaError_t launch_shard_state(const float4* part_f, const int* part_i, int rows, int grid,
                               float* state, cudaStream_t st) {
  shard_state_kernel<<<static_cast<unsigned>((rows + 7) / 8), 256, 0, st>>>(part_f, part_i, rows,
                                                                            grid, state);
  return cudaGetLastError();
}

cudaError_t launch_merge_shards(const float* states, int shards, int rows, int V, float inv_log_v,
                                float* conf, float* entropy, float* ent_norm, float* gap,
                                int* argmax, int* status, cudaStream_t st) {
  merge_shards_kernel<<<static_cast<unsigned>((rows + 7) / 8), 256, 0, st>>>(
      states, shards, rows, V, inv_log_v, conf, entropy, ent_norm, gap, argmax, status);
  return cudaGetLastError();
}

cudaError_t decide_configure() {
  return cudaFuncSetAttribute(decide_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(sizeof(Smem) + 16));
}

cudaError_t launch_decide(const DecideParams& p, cudaStream_t st) {
  if (p.B <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(p.B * kDecideCluster, 1, 1);
  cfg.blockDim = dim3(kDecideThreads, 1, 1);
  cfg.dynamicSmemBytes = sizeof(Smem) + 16;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, decide_kernel, p);
}

cudaError_t launch_fold_tok(const __nv_bfloat16* w_tok, const __nv_bfloat16* w_emb, float* table,
                            int V, int d_base, cudaStream_t st) {
  fold_tok_kernel<<<(V + 63) / 64, 256, 0, st>>>(w_tok, w_emb, table, V, d_base);
  return cudaGetLastError();
}

}  // namespace ebd
