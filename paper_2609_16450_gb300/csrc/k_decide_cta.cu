// The EB decision with one CTA per sequence, for windows of up to 32 rows
// (App. E, algorithm "Inference with LBS Block Selection and LPS Parallel
// Commit"; the same steps and arithmetic as the cluster kernel, k_decide.cu):
//   1. merge the LM-head partial states of each window row into
//      kappa, H, H~ = H / ln|V|, Delta and x_hat (App. B, Sec. 5.1, Sec. 5.2);
//   2. with no active block and |M| > L_min: the LBS router (Sec. 5.1,
//      App. C.1) over the masked rows, then EOS removal, MaxGapFilter and the
//      min-tokens fallback; with |M| <= L_min: B = M;
//   3. the LPS router (Sec. 5.2, App. D.1) over the masked rows of B;
//   4. union accept, anti-stall fallback, parallel commit, block resolution.
//
// Why one CTA.  The kernel is a programmatic dependent of the LM head, whose
// grid leaves SMs free at these sizes (142 CTAs on 152 SMs at 32 rows of a
// 126,464-token vocabulary).  A single CTA is placed on a free SM as soon as
// the LM head releases its dependents, long before the LM head completes; an
// 8-CTA cluster needs 8 free SMs in one GPC and is placed only as the LM
// head drains.  With `warm` set (the host sets it when the LM head leaves
// enough SMs free for every sequence), the CTA first runs the whole decision
// on a stand-in window (results discarded, nothing written to global
// memory): that brings the kernel's code into this SM's instruction caches
// and the router weights into L2 (loaded with an evict-last policy; the LM
// head streams W_lm evict-first), and then waits for the LM head's grid.
//
// LBS products on the tcgen05 tensor cores.  On one SM the products are
// bound by shared-memory reads: mma.sync tiles re-read the activations for
// every 8 outputs.  Here the weights are the A operand (M = 128 output
// features per tile, read once by the tensor core) and the activations the B
// operand, N = 64 rows: the bf16 high parts of the (up to 32) rows and then
// their low parts, so that one MMA computes W hi and W lo side by side in
// TMEM and the epilogue adds the halves (x = hi + lo to ~16 mantissa bits,
// the precision of the cluster kernel's products).  The weight tiles (560 KB
// in all) stream in 16 KB chunks through a ring of kSlots slots in the order
// the phases consume them (rcta layout in router_image.h); thread 0 refills
// the ring at the barrier that ends each phase and issues the MMAs.  The
// attention (4 heads of 32 over <= 32 rows) and the LPS router stay on
// mma.sync.
#include <climits>

#include "decide_common.cuh"

namespace ebd {

namespace {

using namespace rimg::rcta;

constexpr int WC = kCtaWindow;
constexpr int kSlots = 6;  // ring slots of one chunk each
constexpr uint32_t kChunkBytes = kChunkElems * 2u;
constexpr uint64_t kWaitNs = 1000ull * 1000 * 1000;
constexpr uint32_t kTmemCols = 256;  // three 64-column accumulators at most
constexpr int kBBox = 8192;          // bytes of one 64-column box of a B operand

// activation pool (floats), LBS phase; the LPS router's layout (L_*) overlays it.
// B operands ([64][K] bf16, K-major, 128-byte swizzle) start on 1024 bytes.
constexpr int P_BZ = 0;                     // B, K = 128: z (hi | lo)
constexpr int P_BX = P_BZ + 2 * kBBox / 4;  // B, K = 128: [e; t], then the attention output
constexpr int P_R = P_BX + 2 * kBBox / 4;   // B, K = 64: F_ent hidden | B, K = 128 each: q, k, v
                                            // | B, K = 256: FFN hidden
constexpr int P_Z = P_R + 6 * kBBox / 4;    // fp32 [32][132]: ent2 output, then the residual z
constexpr int C_POOL = P_Z + WC * LDZ;
static_assert(L_PROB + W <= C_POOL, "LPS pool layout");
static_assert(rimg::rcta::kPosRows >= WC, "E_pos rows");
// ring entries of one launch: a stand-in run and the real one, each the LBS
// chunks, pads and the LPS chunks
constexpr int kSeqMax = 2 * (kChunks + kSlots);

struct __align__(1024) CtaSmem {
  __nv_bfloat16 ring[kSlots][kChunkElems];
  float pool[C_POOL];
  float v[S_ELEMS];
  float f_conf[WC], f_ent[WC], f_gap[WC], f_O[WC], f_p[WC];
  int f_arg[WC], f_pos[WC], f_tok[WC], Mrows[WC], Brows[WC], BMrows[WC];
  uint8_t f_mask[WC], f_ib[WC], f_acc[WC], f_bad[WC];
  DecideParams p;      // the launch's parameters, for the out-of-line phases
  short seq[kSeqMax];  // chunk of each ring entry, in consumption order; -1: a pad
  int nseq, issued, consumed, wait_err;
  int nM, nBM, meta_b, meta_s, n_rows;
  int r0, n_real, meta_b_real, meta_s_real, bad_seq, lbs_real;
  uint32_t tmem;
  uint64_t full[kSlots];
  uint64_t vbar, mma_bar;
};
static_assert(sizeof(CtaSmem) <= 232448, "dynamic shared memory of one CTA");
static_assert(offsetof(CtaSmem, pool) % 1024 == 0, "B operands on 1024-byte boundaries");

// The CTA's dynamic shared memory.  Functions reach it through this symbol,
// not through a pointer argument, so that their accesses compile to
// shared-memory instructions even out of line.
extern __shared__ __align__(1024) uint8_t cta_dsmem[];
__device__ __forceinline__ CtaSmem& cta_smem() { return *reinterpret_cast<CtaSmem*>(cta_dsmem); }

// Orders this thread's earlier shared-memory accesses (generic proxy) before
// later accesses by the async proxy (bulk copies, tcgen05.mma operand reads).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void bulk_copy_keep(void* smem_dst, const void* gsrc, uint32_t bytes,
                                               uint64_t* bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
      "[%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(smem_dst)),
      "l"(gsrc), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

// Thread 0: issues ring entries while a slot is free.  Entry i goes to slot
// i % kSlots once entry i - kSlots has been consumed; a pad completes its
// slot's phase with a plain arrive.  Called after the barrier that ends the
// phase which consumed the entries below sm.consumed.
__device__ void ring_fill(const __nv_bfloat16* img) {
  CtaSmem& sm = cta_smem();
  if (sm.issued >= sm.nseq || sm.issued >= sm.consumed + kSlots) return;
  fence_proxy_async_smem();  // the freed slots' earlier ordinary reads (LPS weights)
  const uint64_t pol = l2_policy_evict_last();
  while (sm.issued < sm.nseq && sm.issued < sm.consumed + kSlots) {
    const int i = sm.issued++;
    uint64_t* bar = &sm.full[i % kSlots];
    const int c = sm.seq[i];
    if (c < 0) {
      mbar_arrive(bar);
      continue;
    }
    mbar_arrive_expect_tx(bar, kChunkBytes);
    bulk_copy_keep(sm.ring[i % kSlots], img + static_cast<size_t>(c) * kChunkElems, kChunkBytes, bar,
                   pol);
  }
}

// ring entries [q, q + k) have landed
__device__ __forceinline__ void ring_wait(CtaSmem& sm, int q, int k) {
  for (int i = q; i < q + k; ++i)
    if (!mbar_wait(&sm.full[i % kSlots], static_cast<uint32_t>(i / kSlots) & 1u, kWaitNs, nullptr))
      sm.wait_err = 1;
}

// after the barrier that ends a phase: the entries below q are consumed
__device__ __forceinline__ void ring_release(CtaSmem& sm, int q) {
  if (threadIdx.x == 0) {
    sm.consumed = q;
    ring_fill(sm.p.w.cta_w);
  }
}

// ------------------------------------------------------------------ B operands
// A B operand holds activation rows as [64][K] bf16: row r < 32 the high part
// of activation row r, row 32 + r its low part; K-major, 64-column boxes of
// 8 KB, 128-byte swizzle (16-byte chunk c of a row at chunk c ^ (row & 7)).
__device__ __forceinline__ uint32_t b_off(int r, int k) {
  const int w = k & 63;
  return static_cast<uint32_t>((k >> 6) * kBBox + r * 128 + ((((w >> 3) ^ (r & 7)) << 4) | ((w & 7) << 1)));
}
// (x, y) as columns k, k + 1 (k even) of activation row r
__device__ __forceinline__ void b_store2(uint8_t* buf, int r, int k, float x, float y) {
  uint32_t hi, lo;
  split_bf16x2(x, y, hi, lo);
  *reinterpret_cast<uint32_t*>(buf + b_off(r, k)) = hi;
  *reinterpret_cast<uint32_t*>(buf + b_off(r + 32, k)) = lo;
}

// One unit of the LBS attention: query rows [16 qt, 16 qt + 16) of head h
// (width 32) over all n <= 32 keys, output columns [16 hf, 16 hf + 16) of
// the head: softmax(q k^T / sqrt(32)) v on the tensor cores, with q, k, v
// (B-operand layout, high and low parts) read by ldmatrix and three
// products per pair (hi hi, hi lo, lo hi).  All keys fit in two 16-key
// blocks, so the row max is taken over every score before the
// exponentials; v rows from n up to the block end must be finite (zeros).
// The result goes to columns 32 h + 16 hf .. + 16 of the B operand `out`.
__device__ __forceinline__ void lbs_attn_unit(const uint8_t* qb, const uint8_t* kb_, const uint8_t* vb,
                                              int n, int qt, int h, int hf, uint8_t* out) {
  const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const int mi = lane >> 3, rr = lane & 7;
  constexpr uint32_t kLo = 32 * 128;  // bytes from a row's high part to its low part
  const float scale = 0.17677669529663687f;  // 1/sqrt(32)
  uint32_t qh[2][4], ql[2][4];
#pragma unroll
  for (int ks = 0; ks < 2; ++ks) {
    const uint32_t a = smem_u32(qb) + b_off(16 * qt + (mi & 1) * 8 + rr, 32 * h + 16 * ks + (mi >> 1) * 8);
    ldsm_x4(a, qh[ks][0], qh[ks][1], qh[ks][2], qh[ks][3]);
    ldsm_x4(a + kLo, ql[ks][0], ql[ks][1], ql[ks][2], ql[ks][3]);
  }
  const int nkb = (n + 15) >> 4;  // 1 or 2
  float s[2][2][4];               // [key block][8-key half][fragment]
#pragma unroll
  for (int kb = 0; kb < 2; ++kb) {
#pragma unroll
    for (int hb = 0; hb < 2; ++hb) {
      float a[4] = {0.f, 0.f, 0.f, 0.f};
      if (kb < nkb) {
        // keys 16 kb + 8 hb + (lane & 7); matrices: dims 0-7, 8-15, 16-23, 24-31 of the head
        const uint32_t ka = smem_u32(kb_) + b_off(16 * kb + 8 * hb + rr, 32 * h + 8 * mi);
        uint32_t kh[4], kl[4];
        ldsm_x4(ka, kh[0], kh[1], kh[2], kh[3]);
        ldsm_x4(ka + kLo, kl[0], kl[1], kl[2], kl[3]);
        mma_bf16(a, qh[0], kh[0], kh[1]);
        mma_bf16(a, qh[0], kl[0], kl[1]);
        mma_bf16(a, ql[0], kh[0], kh[1]);
        mma_bf16(a, qh[1], kh[2], kh[3]);
        mma_bf16(a, qh[1], kl[2], kl[3]);
        mma_bf16(a, ql[1], kh[2], kh[3]);
      }
      const int c = 16 * kb + 8 * hb + 2 * t;
      s[kb][hb][0] = c < n ? a[0] * scale : -INFINITY;
      s[kb][hb][1] = c + 1 < n ? a[1] * scale : -INFINITY;
      s[kb][hb][2] = c < n ? a[2] * scale : -INFINITY;
      s[kb][hb][3] = c + 1 < n ? a[3] * scale : -INFINITY;
    }
  }
  float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
  for (int kb = 0; kb < 2; ++kb)
#pragma unroll
    for (int hb = 0; hb < 2; ++hb) {
      m0 = fmaxf(m0, fmaxf(s[kb][hb][0], s[kb][hb][1]));
      m1 = fmaxf(m1, fmaxf(s[kb][hb][2], s[kb][hb][3]));
    }
  m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, 1));
  m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, 2));
  m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, 1));
  m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, 2));  // finite: key 0 is valid
  float l0 = 0.f, l1 = 0.f;
#pragma unroll
  for (int kb = 0; kb < 2; ++kb)
#pragma unroll
    for (int hb = 0; hb < 2; ++hb) {
      s[kb][hb][0] = expf(s[kb][hb][0] - m0);
      s[kb][hb][1] = expf(s[kb][hb][1] - m0);
      s[kb][hb][2] = expf(s[kb][hb][2] - m1);
      s[kb][hb][3] = expf(s[kb][hb][3] - m1);
      l0 += s[kb][hb][0] + s[kb][hb][1];
      l1 += s[kb][hb][2] + s[kb][hb][3];
    }
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  float o[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
  for (int kb = 0; kb < 2; ++kb) {
    if (kb >= nkb) break;
    uint32_t ph[4], pl[4];
    split_bf16x2(s[kb][0][0], s[kb][0][1], ph[0], pl[0]);
    split_bf16x2(s[kb][0][2], s[kb][0][3], ph[1], pl[1]);
    split_bf16x2(s[kb][1][0], s[kb][1][1], ph[2], pl[2]);
    split_bf16x2(s[kb][1][2], s[kb][1][3], ph[3], pl[3]);
    // keys 16 kb + (lane & 7) + 8 ((lane >> 3) & 1); columns 16 hf + 8 (lane >> 4) of the head
    const uint32_t va = smem_u32(vb) + b_off(16 * kb + rr + 8 * (mi & 1), 32 * h + 16 * hf + 8 * (mi >> 1));
    uint32_t vh[4], vl[4];
    ldsm_x4_t(va, vh[0], vh[1], vh[2], vh[3]);
    ldsm_x4_t(va + kLo, vl[0], vl[1], vl[2], vl[3]);
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      mma_bf16(o[i], ph, vh[2 * i], vh[2 * i + 1]);
      mma_bf16(o[i], ph, vl[2 * i], vl[2 * i + 1]);
      mma_bf16(o[i], pl, vh[2 * i], vh[2 * i + 1]);
    }
  }
  const float i0 = 1.0f / l0, i1 = 1.0f / l1;
  const int r_lo = 16 * qt + g, r_hi = r_lo + 8;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int c = 32 * h + 16 * hf + 8 * i + 2 * t;
    if (r_lo < n) b_store2(out, r_lo, c, o[i][0] * i0, o[i][1] * i0);
    if (r_hi < n) b_store2(out, r_hi, c, o[i][2] * i1, o[i][3] * i1);
  }
}

// LayerNorm (eps 1e-5) over DIM (64 or 128) features of rows j < n (8 lanes
// per row, lane q holding columns 4q + 32c); the result goes to columns
// kofs.. of the B operand b and, if dst is set, to dst (which may be src).
template <int DIM>
__device__ __forceinline__ void ln_rows_b(const float* src, int lds, float* dst, int ldd, uint8_t* b,
                                          int kofs, int n, const float* g, const float* bb) {
  constexpr int PER = DIM / 32;
  const int q = threadIdx.x & 7;
#pragma unroll 1
  for (int j0 = 0; j0 < n; j0 += (blockDim.x >> 3)) {
    const int j = j0 + (threadIdx.x >> 3);
    const bool ok = j < n;
    float4 v[PER];
    float s = 0.f;
#pragma unroll
    for (int c = 0; c < PER; ++c) {
      v[c] = ok ? *reinterpret_cast<const float4*>(src + j * lds + 4 * q + 32 * c)
                : make_float4(0.f, 0.f, 0.f, 0.f);
      s += (v[c].x + v[c].y) + (v[c].z + v[c].w);
    }
    const float mean = group8_sum(s) * (1.0f / DIM);
    float var = 0.f;
#pragma unroll
    for (int c = 0; c < PER; ++c) {
      const float a0 = v[c].x - mean, a1 = v[c].y - mean, a2 = v[c].z - mean, a3 = v[c].w - mean;
      var += (a0 * a0 + a1 * a1) + (a2 * a2 + a3 * a3);
    }
    const float inv = rsqrtf(group8_sum(var) * (1.0f / DIM) + 1e-5f);
    if (ok) {
#pragma unroll
      for (int c = 0; c < PER; ++c) {
        const int o = 4 * q + 32 * c;
        const float4 gg = *reinterpret_cast<const float4*>(g + o);
        const float4 be = *reinterpret_cast<const float4*>(bb + o);
        const float4 y = make_float4((v[c].x - mean) * inv * gg.x + be.x, (v[c].y - mean) * inv * gg.y + be.y,
                                     (v[c].z - mean) * inv * gg.z + be.z, (v[c].w - mean) * inv * gg.w + be.w);
        if (dst != nullptr) *reinterpret_cast<float4*>(dst + j * ldd + o) = y;
        uint32_t h0, l0, h1, l1;
        split_bf16x2(y.x, y.y, h0, l0);
        split_bf16x2(y.z, y.w, h1, l1);
        *reinterpret_cast<uint2*>(b + b_off(j, kofs + o)) = make_uint2(h0, h1);
        *reinterpret_cast<uint2*>(b + b_off(j + 32, kofs + o)) = make_uint2(l0, l1);
      }
    }
  }
}

// ------------------------------------------------------------------ tcgen05 products
// Thread 0: the accumulator of tile t (TMEM columns 64 t, t < T) = A_t B^T
// over K = 64 nkb, where A_t's K-boxes are ring entries q + t nkb + kb and
// B is the operand at b; completion arrives on sm.mma_bar.
__device__ __forceinline__ void mma_issue(const CtaSmem& sm, int q, int T, int nkb, const uint8_t* b) {
  tc_fence_after();
  const uint32_t hi = static_cast<uint32_t>(umma_desc_sw128(0) >> 32);
  constexpr uint32_t idesc = umma_idesc_bf16(128, 64);
  const uint32_t b_lo = static_cast<uint32_t>(umma_desc_sw128(smem_u32(b)));
#pragma unroll 1
  for (int t = 0; t < T; ++t)
#pragma unroll 1
    for (int kb = 0; kb < nkb; ++kb) {
      const uint32_t a_lo =
          static_cast<uint32_t>(umma_desc_sw128(smem_u32(sm.ring[(q + t * nkb + kb) % kSlots])));
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        umma_bf16_lo(sm.tmem + 64u * t, a_lo + 2u * kk,
                     b_lo + static_cast<uint32_t>(kb * (kBBox >> 4)) + 2u * kk, hi, idesc,
                     (kb | kk) != 0 ? 1u : 0u);
    }
  umma_commit(const_cast<uint64_t*>(&sm.mma_bar));
}

// every thread: the MMAs of the phase with this parity have completed
__device__ __forceinline__ void mma_wait(CtaSmem& sm, uint32_t parity) {
  if (!mbar_wait(&sm.mma_bar, parity, kWaitNs, nullptr)) sm.wait_err = 1;
  tc_fence_after();
}

// The epilogue of T accumulator tiles: epi(r, f, x, y) for the output
// features f and f + 1 (f even, < fmax, a multiple of 64) of row r < n,
// each value W hi + W lo of that row (columns r and 32 + r).  Warpgroup g
// takes the (tile, 8-row group) units g, g + 4, ...; a warp reads its TMEM
// lane quadrant (a lane one feature, 8 rows), then lanes 2k and 2k + 1 swap
// halves so that each holds 4 rows of the feature pair: stores of two
// adjacent bf16 or fp32 values.
template <class Epi>
__device__ __forceinline__ void mma_epilogue(const CtaSmem& sm, int T, int n, int fmax, Epi epi) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quad = warp & 3;
  const int ngroups = (n + 7) >> 3;
#pragma unroll 1
  for (int u = warp >> 2; u < T * 4; u += (blockDim.x >> 7)) {
    const int t = u >> 2, g8 = u & 3;
    if (g8 >= ngroups) continue;
    const uint32_t ta = sm.tmem + (static_cast<uint32_t>(32 * quad) << 16) + 64u * t + 8u * g8;
    uint32_t rh[8], rl[8];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%16];\n"
        "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%8,%9,%10,%11,%12,%13,%14,%15}, [%17];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(rh[0]), "=r"(rh[1]), "=r"(rh[2]), "=r"(rh[3]), "=r"(rh[4]), "=r"(rh[5]), "=r"(rh[6]),
          "=r"(rh[7]), "=r"(rl[0]), "=r"(rl[1]), "=r"(rl[2]), "=r"(rl[3]), "=r"(rl[4]), "=r"(rl[5]),
          "=r"(rl[6]), "=r"(rl[7])
        : "r"(ta), "r"(ta + 32u)
        : "memory");
    const int f = 128 * t + 32 * quad + lane;
    if (f >= fmax) continue;  // the whole warp: fmax is a multiple of 64
    const bool odd = (lane & 1) != 0;
    const int fe = f & ~1;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float lo_row = __uint_as_float(rh[i]) + __uint_as_float(rl[i]);          // row i
      const float hi_row = __uint_as_float(rh[4 + i]) + __uint_as_float(rl[4 + i]);  // row 4 + i
      const float got = __shfl_xor_sync(0xffffffffu, odd ? lo_row : hi_row, 1);
      // even lane: row i of features (f, f + 1); odd lane: row 4 + i of (f - 1, f)
      const int r = 8 * g8 + (odd ? 4 + i : i);
      if (r < n) epi(r, fe, odd ? got : lo_row, odd ? hi_row : got);
    }
  }
}

// The LBS router (Sec. 5.1, App. C.1) over the n = |M| masked rows
// (sm.Mrows): entropy branch F_ent, token branch, fusion with E_pos, two
// post-norm encoder layers (4 heads of width 32, FFN 256, GELU), head
// Linear(128 -> 1); the logit of masked row j goes to f_O[Mrows[j]].
// Consumes ring entries [q, q + C_LPS) and ten MMA phases (an even number:
// every call starts at mbarrier parity 0).
__device__ __noinline__ void lbs_forward(int n, int q) {
  CtaSmem& sm = cta_smem();
  const DecideParams& p = sm.p;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nwarps = blockDim.x >> 5;
  float* P = sm.pool;
  const float* Vv = sm.v;
  uint8_t* bz = reinterpret_cast<uint8_t*>(P + P_BZ);
  uint8_t* bx = reinterpret_cast<uint8_t*>(P + P_BX);
  uint8_t* br = reinterpret_cast<uint8_t*>(P + P_R);  // F_ent hidden, q | k | v, FFN hidden
  uint8_t* bq = br;
  uint8_t* bk = br + 2 * kBBox;
  uint8_t* bv = br + 4 * kBBox;
  float* Z = P + P_Z;
  const __nv_bfloat16* pos = reinterpret_cast<const __nv_bfloat16*>(Vv + S_POS);
  uint32_t ph = 0;

  // 1. entropy branch, first layer -> B (K = 64); the token branch's gathers
  // from the folded table are issued first and stored later, hiding their latency
  static_assert(kCtaThreads * 2 >= WC * 32, "token-branch items per thread");
  float2 tv[2];
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const int it = tid + k * kCtaThreads;
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
    b_store2(br, j, o, gelu(fmaf(Vv[S_ENT1W + o], h, Vv[S_ENT1B + o])),
             gelu(fmaf(Vv[S_ENT1W + o + 1], h, Vv[S_ENT1B + o + 1])));
  }
  fence_proxy_async_smem();
  if (tid == 0) ring_wait(sm, q, 3);
  __syncthreads();
  // 2. ent2 (64 outputs) into z's region
  if (tid == 0) mma_issue(sm, q, 1, 1, br);
  mma_wait(sm, ph);
  ph ^= 1u;
  mma_epilogue(sm, 1, n, 64, [&](int r, int f, float x, float y) {
    *reinterpret_cast<float2*>(Z + r * LDZ + f) = make_float2(x + Vv[S_ENT2B + f], y + Vv[S_ENT2B + f + 1]);
  });
  tc_fence_before();
  __syncthreads();
  // 3. e = LayerNorm(ent2) -> columns 0..63 of [e; t], t -> 64..127
  ln_rows_b<64>(Z, LDZ, nullptr, 0, bx, 0, n, Vv + S_ENTLNG, Vv + S_ENTLNB);
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const int it = tid + k * kCtaThreads;
    if (it < n * 32) {
      const int o = 2 * (it & 31);
      b_store2(bx, it >> 5, 64 + o, tv[k].x + Vv[S_TOKB + o], tv[k].y + Vv[S_TOKB + o + 1]);
    }
  }
  fence_proxy_async_smem();
  __syncthreads();
  // 4. fusion: z = W_combine [e; t] + b + E_pos[j], and z as the first QKV input
  if (tid == 0) mma_issue(sm, q + 1, 1, 2, bx);
  mma_wait(sm, ph);
  ph ^= 1u;
  mma_epilogue(sm, 1, n, 128, [&](int r, int f, float x, float y) {
    const float2 pe = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(pos + r * 128 + f));
    const float z0 = x + Vv[S_COMBB + f] + pe.x, z1 = y + Vv[S_COMBB + f + 1] + pe.y;
    *reinterpret_cast<float2*>(Z + r * LDZ + f) = make_float2(z0, z1);
    b_store2(bz, r, f, z0, z1);
  });
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  q += 3;
  ring_release(sm, q);
  // 5. two post-norm encoder layers
  const int mtq = (n + 15) >> 4;
#pragma unroll 1
  for (int l = 0; l < 2; ++l) {
    const float* Vl = Vv + S_LAYER0 + l * S_LAYER_STRIDE;
    if (tid == 0) {
      ring_wait(sm, q, 6);
      mma_issue(sm, q, 3, 2, bz);
    }
    mma_wait(sm, ph);
    ph ^= 1u;
    mma_epilogue(sm, 3, n, 384, [&](int r, int f, float x, float y) {
      b_store2(f < 128 ? bq : (f < 256 ? bk : bv), r, f & 127, x + Vl[SL_QKVB + f], y + Vl[SL_QKVB + f + 1]);
    });
    // v rows n..31: zeros (the products with key blocks that end past n read them)
#pragma unroll 1
    for (int it = tid; it < (WC - n) * 32; it += blockDim.x) {
      const int r = n + (it >> 5), c = 8 * (it & 15), lo = (it >> 4) & 1;
      *reinterpret_cast<uint4*>(bv + b_off(r + 32 * lo, c)) = make_uint4(0u, 0u, 0u, 0u);
    }
    tc_fence_before();
    __syncthreads();
    q += 6;
    ring_release(sm, q);
#pragma unroll 1
    for (int u = warp; u < 4 * mtq * 2; u += nwarps)
      lbs_attn_unit(bq, bk, bv, n, (u >> 1) % mtq, u / (2 * mtq), u & 1, bx);
    fence_proxy_async_smem();
    if (tid == 0) ring_wait(sm, q, 2);
    __syncthreads();
    // output projection + residual, in place into z
    if (tid == 0) mma_issue(sm, q, 1, 2, bx);
    mma_wait(sm, ph);
    ph ^= 1u;
    mma_epilogue(sm, 1, n, 128, [&](int r, int f, float x, float y) {
      float2* z = reinterpret_cast<float2*>(Z + r * LDZ + f);
      const float2 zz = *z;
      *z = make_float2(zz.x + (x + Vl[SL_OUTB + f]), zz.y + (y + Vl[SL_OUTB + f + 1]));
    });
    tc_fence_before();
    __syncthreads();
    q += 2;
    ring_release(sm, q);
    ln_rows_b<128>(Z, LDZ, Z, LDZ, bz, 0, n, Vl + SL_LN1G, Vl + SL_LN1B);
    fence_proxy_async_smem();
    if (tid == 0) ring_wait(sm, q, 4);
    __syncthreads();
    // FFN: hidden = GELU(W1 z + b1) as a B operand (K = 256), z += W2 hidden + b2
    if (tid == 0) mma_issue(sm, q, 2, 2, bz);
    mma_wait(sm, ph);
    ph ^= 1u;
    mma_epilogue(sm, 2, n, 256, [&](int r, int f, float x, float y) {
      b_store2(br, r, f, gelu(x + Vl[SL_FF1B + f]), gelu(y + Vl[SL_FF1B + f + 1]));
    });
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    q += 4;
    ring_release(sm, q);
    if (tid == 0) {
      ring_wait(sm, q, 4);
      mma_issue(sm, q, 1, 4, br);
    }
    mma_wait(sm, ph);
    ph ^= 1u;
    mma_epilogue(sm, 1, n, 128, [&](int r, int f, float x, float y) {
      float2* z = reinterpret_cast<float2*>(Z + r * LDZ + f);
      const float2 zz = *z;
      *z = make_float2(zz.x + (x + Vl[SL_FF2B + f]), zz.y + (y + Vl[SL_FF2B + f + 1]));
    });
    tc_fence_before();
    __syncthreads();
    q += 4;
    ring_release(sm, q);
    ln_rows_b<128>(Z, LDZ, Z, LDZ, bz, 0, n, Vl + SL_LN2G, Vl + SL_LN2B);
    fence_proxy_async_smem();
    __syncthreads();
  }
  // 6. head Linear(128 -> 1)
#pragma unroll 1
  for (int j = warp; j < n; j += nwarps) {
    float a = 0.f;
#pragma unroll
    for (int c = 0; c < 4; ++c) a += Z[j * LDZ + lane + 32 * c] * Vv[S_HEADW + lane + 32 * c];
    a = warp_sum(a) + Vv[S_HEADB];
    if (lane == 0) sm.f_O[sm.Mrows[j]] = a;
  }
  __syncthreads();
}

// Steps 2-4 of the decision for the window in shared memory (f_*, Mrows,
// nM, meta_b/meta_s), from ring entry q on; `lbs`: the LBS runs (the ring
// holds its chunks).  Not inlined: the stand-in run and the real one execute
// the same instructions.
__device__ __noinline__ void decide_window(int q, bool lbs) {
  CtaSmem& sm = cta_smem();
  const DecideParams& p = sm.p;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nr = sm.n_rows, nM = sm.nM;
  if (lbs) {
    lbs_forward(nM, q);
    q += C_LPS;
  }

  // ---------------------------------------------------------------- block selection
  if (warp == 0) {
    if (p.mode != EBD_DECODE_EB) {
      // baselines: the window is the active fixed block; no block state
    } else if (sm.meta_s == 0) {
      for (int j = lane; j < nr; j += 32) sm.f_ib[j] = 0;
      __syncwarp();
      int nB = 0;
      if (!lbs) {  // |M| <= L_min: B = M
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

  // ---------------------------------------------------------------- LPS
  const int nBM = sm.nBM;
  if (p.lps_enabled) {
    while (sm.seq[q] < 0) ++q;  // pads that keep the three LPS chunks in consecutive slots
    ring_wait(sm, q, LPS_CHUNKS);
    if (nBM > 0) {
      float* feats = sm.pool + L_FEAT;
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
      lps_forward(sm.pool, nBM, sm.ring[q % kSlots], sm.v + S_LPS, 0, 8);
      const float* prob = sm.pool + L_PROB;
#pragma unroll 1
      for (int i = tid; i < nBM; i += blockDim.x) sm.f_p[sm.BMrows[i]] = prob[i];
    }
    __syncthreads();
    q += LPS_CHUNKS;
    ring_release(sm, q);
  }

  // ---------------------------------------------------------------- accept and commit
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
      if (lane == 0 && bj < nr) sm.f_acc[bj] = 1;
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
}

// masked set M of the window in shared memory (warp 0)
__device__ __noinline__ void masked_set() {
  CtaSmem& sm = cta_smem();
  const int lane = threadIdx.x & 31;
  const int nr = sm.n_rows;
  int base = 0;
  for (int j0 = 0; j0 < nr; j0 += 32) {
    const int j = j0 + lane;
    const bool m = j < nr && sm.f_mask[j];
    const uint32_t bal = __ballot_sync(0xffffffffu, m);
    if (m) sm.Mrows[base + __popc(bal & ((1u << lane) - 1u))] = j;
    base += __popc(bal);
  }
  if (lane == 0) sm.nM = base;
}

}  // namespace

__global__ void __launch_bounds__(kCtaThreads, 1) decide_cta_kernel(const DecideParams p) {
  CtaSmem& sm = cta_smem();
  const int seq = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // a kernel launched after this one as a programmatic dependent (the window
  // attention, which shares no data with the decision) may start on the SMs
  // this grid leaves free
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  // the B operands' 128-byte swizzle is laid out from a 1024-byte boundary
  if ((smem_u32(cta_dsmem) & 1023u) != 0u) {
    if (tid == 0) atomicCAS(p.status, 0, EBD_ERR_UNSUPPORTED);
    return;
  }
  const bool eb = p.mode == EBD_DECODE_EB;
  const bool warm = p.warm && eb;

  // ---------------------------------------------------------------- setup
  // The decode state of this step was written by kernels that completed
  // before the LM head released this grid: it is read now.  Whether the LBS
  // runs (no active block, |M| > L_min) fixes the ring's chunk sequence.
  if (tid == 32) sm.p = p;
  if (warp == 0) {
    tmem_alloc(&sm.tmem, kTmemCols);  // the whole warp; this CTA fills its SM
    int r0 = 0, nr = 0, bad = 0;
    if (lane == 0) {
      for (int s = 0; s < kSlots; ++s) mbar_init(&sm.full[s], 1);
      mbar_init(&sm.vbar, 1);
      mbar_init(&sm.mma_bar, 1);
      fence_mbar_init();
      mbar_arrive_expect_tx(&sm.vbar, S_ELEMS * 4u);
      bulk_copy(sm.v, p.w.cta_vec, S_ELEMS * 4u, &sm.vbar);
      r0 = p.cu_rows[seq];
      const int r1 = p.cu_rows[seq + 1];
      nr = r1 - r0;
      if (p.cu_rows[p.B] != p.rows_expected || nr < 0 || nr > WC || r0 < 0) {
        bad = 1;
        atomicCAS(p.status, 0, EBD_ERR_INVALID_ARG);
      }
      if (bad) nr = 0;
      sm.meta_b_real = p.blk_meta[2 * seq];
      sm.meta_s_real = p.blk_meta[2 * seq + 1];
    }
    r0 = __shfl_sync(0xffffffffu, r0, 0);
    nr = __shfl_sync(0xffffffffu, nr, 0);
    const bool m = lane < nr && in_bounds(r0 + lane, p.rows_expected, p.status) && p.mask[r0 + lane];
    const int nm = __popc(__ballot_sync(0xffffffffu, m));
    if (lane == 0) {
      sm.r0 = r0;
      sm.n_real = nr;
      sm.bad_seq = bad;
      const int lbs = eb && sm.meta_s_real == 0 && nm > p.l_min;
      sm.lbs_real = lbs;
      int n = 0;
      auto add_lbs = [&]() {
        for (int c = 0; c < C_LPS; ++c) sm.seq[n++] = static_cast<short>(c);
      };
      auto add_lps = [&]() {
        while (n % kSlots > kSlots - LPS_CHUNKS) sm.seq[n++] = -1;
        for (int c = 0; c < LPS_CHUNKS; ++c) sm.seq[n++] = static_cast<short>(C_LPS + c);
      };
      if (warm) {
        add_lbs();
        if (p.lps_enabled) add_lps();
      }
      if (lbs) add_lbs();
      if (p.lps_enabled) add_lps();
      sm.seq[n] = 0;  // a sentinel for the pad scan
      sm.nseq = n;
      sm.issued = 0;
      sm.consumed = 0;
      sm.wait_err = 0;
      ring_fill(p.w.cta_w);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (!mbar_wait(&sm.vbar, 0, kWaitNs, nullptr)) sm.wait_err = 1;
  int q = 0;

  // ---------------------------------------------------------------- stand-in run
  if (warm) {
    for (int j = tid; j < WC; j += blockDim.x) {
      sm.f_mask[j] = 1;
      sm.f_ib[j] = 0;
      sm.f_tok[j] = 0;
      sm.f_pos[j] = j;
      sm.f_acc[j] = 0;
      sm.f_O[j] = __int_as_float(0x7fc00000);
      sm.f_p[j] = __int_as_float(0x7fc00000);
      sm.f_conf[j] = 0.25f + 0.02f * static_cast<float>(j);
      sm.f_ent[j] = 0.5f - 0.01f * static_cast<float>(j);
      sm.f_gap[j] = 0.1f;
      sm.f_arg[j] = j % p.V;
      sm.f_bad[j] = 0;
    }
    if (tid == 0) {
      sm.n_rows = WC;
      sm.meta_b = 0;
      sm.meta_s = 0;
    }
    __syncthreads();
    if (warp == 0) masked_set();
    __syncthreads();
    decide_window(q, true);
    q += C_LPS;
    if (p.lps_enabled) {
      while (sm.seq[q] < 0) ++q;
      q += LPS_CHUNKS;
    }
  }

  // ---------------------------------------------------------------- the window's state
  const int r0 = sm.r0, nr = sm.n_real;
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
  if (tid == 0) {
    sm.n_rows = nr;
    sm.meta_b = sm.meta_b_real;
    sm.meta_s = sm.meta_s_real;
  }

  // ---------------------------------------------------------------- 1. statistics
  // the partial states are read only after the LM head's grid has completed
  // and its writes are visible
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
#pragma unroll 1
    for (int j = warp; j < nr; j += (blockDim.x >> 5)) {
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
      for (int c = 0; c < 8; ++c) merge_state(m, s, t, l2, idx, fv[c].x, fv[c].y, fv[c].z, fv[c].w, iv[c]);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float bm = __shfl_xor_sync(0xffffffffu, m, off);
        const float bs = __shfl_xor_sync(0xffffffffu, s, off);
        const float bt = __shfl_xor_sync(0xffffffffu, t, off);
        const float bl = __shfl_xor_sync(0xffffffffu, l2, off);
        const int bi = __shfl_xor_sync(0xffffffffu, idx, off);
        merge_state(m, s, t, l2, idx, bm, bs, bt, bl, bi);
      }
      if (lane == 0) {
        const float conf = 1.0f / s;
        const float ent = logf(s) - t / s;
        const float entn = ent * p.inv_log_v;
        const float gap = (1.0f - expf(l2 - m)) / s;
        const bool bad = !(isfinite(m) && isfinite(s) && isfinite(t) && s >= 1.0f) || idx < 0 ||
                         idx >= p.V;
        const int r = r0 + j;
        if (in_bounds(r, p.rows_expected, p.status)) {
          if (p.conf) p.conf[r] = conf;
          if (p.entropy) p.entropy[r] = ent;
          if (p.ent_norm) p.ent_norm[r] = entn;
          if (p.gap) p.gap[r] = gap;
          if (p.argmax) p.argmax[r] = bad ? -1 : idx;
          if (bad) atomicCAS(p.status, 0, EBD_ERR_NONFINITE);
        }
        sm.f_conf[j] = conf;
        sm.f_ent[j] = entn;
        sm.f_gap[j] = gap;
        sm.f_arg[j] = bad ? -1 : idx;
        sm.f_bad[j] = bad ? 1 : 0;
      }
    }
  }
  __syncthreads();
  if (warp == 0) masked_set();
  __syncthreads();

  // ---------------------------------------------------------------- 2-4. the decision
  decide_window(q, sm.lbs_real != 0);

  // ---------------------------------------------------------------- write back
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
  if (tid == 0) {
    if (!sm.bad_seq) {
      p.blk_meta_out[2 * seq] = sm.meta_b;
      p.blk_meta_out[2 * seq + 1] = sm.meta_s;
    }
    // every issued copy must have landed before the CTA exits (after a
    // timed-out wait, those still in flight; bounded)
    for (int i = sm.consumed; i < sm.issued; ++i)
      if (!mbar_wait(&sm.full[i % kSlots], static_cast<uint32_t>(i / kSlots) & 1u, kWaitNs, nullptr))
        sm.wait_err = 1;
    if (sm.wait_err) atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
  }
  // every MMA has completed (its commit was waited for) and every TMEM load
  // has returned: the columns go back
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(sm.tmem, kTmemCols);
  }
}

cudaError_t decide_cta_configure() {
  return cudaFuncSetAttribute(decide_cta_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(sizeof(CtaSmem)));
}

cudaError_t launch_decide_cta(const DecideParams& p, cudaStream_t st) {
  if (p.B <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(p.B, 1, 1);
  cfg.blockDim = dim3(kCtaThreads, 1, 1);
  cfg.dynamicSmemBytes = sizeof(CtaSmem);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, decide_cta_kernel, p);
}

}  // namespace ebd
