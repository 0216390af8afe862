// Device code shared by the per-sequence decision kernels (k_decide.cu: one
// 8-CTA cluster per sequence; k_decide_cta.cu: one CTA per sequence): the
// hi/lo bf16 activation format, the tensor-core product over it, LayerNorm,
// the merge of LM-head partial states, and the LPS router (Sec. 5.2,
// App. D.1).
#pragma once
#include "internal.h"
#include "ptx.cuh"
#include "router_image.h"

namespace ebd {
namespace {

using namespace rimg;

constexpr int W = kMaxWindow;  // rows per sequence
constexpr int LDZ = 132;       // fp32 residual stream row stride
constexpr int LDH = 136;       // bf16 hi/lo row stride for 128 columns (conflict-free ldmatrix)
constexpr int LDKV = 68;       // fp32 k in [0,32), v in [32,64)
constexpr int LDQ = 36;
constexpr int LDS = 68;

// activation pool, LPS phase (rank 0)
constexpr int L_FEAT = 0;                    // [64][8] features
constexpr int L_Z = 512;                     // [64][36] fp32 residual stream
constexpr int L_YH = L_Z + W * LDQ;          // [64][40] bf16 x2: LayerNorm output
constexpr int L_QKV = L_YH + W * 40;         // [64][100] fp32 q | k | v
constexpr int L_AH = L_QKV + W * 100;        // [64][40] bf16 x2: attention output
constexpr int L_HH = L_AH + W * 40;          // [64][72] bf16 x2: FFN hidden
constexpr int L_PROB = L_HH + W * 72;        // [64]

__device__ __forceinline__ float gelu(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
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

// hi/lo pair of bf16 buffers: hi at base, lo at base + plane (elements)
struct HL {
  __nv_bfloat16* p;
  int ld, plane;
};
// a hi/lo buffer of `rows` rows of stride ld at pool_floats (hi plane first)
__device__ __forceinline__ HL hl_at(float* pool_floats, int ld, int rows = W) {
  return HL{reinterpret_cast<__nv_bfloat16*>(pool_floats), ld, rows * ld};
}
// stores (x, y) as columns (c, c+1) of row j
__device__ __forceinline__ void hl_store2(const HL& h, int j, int c, float x, float y) {
  uint32_t hi, lo;
  split_bf16x2(x, y, hi, lo);
  *reinterpret_cast<uint32_t*>(h.p + j * h.ld + c) = hi;
  *reinterpret_cast<uint32_t*>(h.p + h.plane + j * h.ld + c) = lo;
}

__device__ __forceinline__ void ldsm_x2_t(uint32_t addr, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];"
               : "=r"(r0), "=r"(r1)
               : "r"(addr));
}

// out(j, o) = sum_k A[j][k] Wt[k][o] for j < n, o < Os, A = hi + lo in
// shared memory, Wt bf16 [K][ldw].  Each warp owns 16-row x 8-output tiles:
// with the few rows of a window, narrow tiles spread a product over more
// warps, and the tensor-core work per warp bounds a phase.  The high and low
// parts accumulate in separate chains, summed at the end.  epi(j, o, v0, v1)
// receives the outputs o and o + 1 of row j.  SWZ: Wt holds its 16-byte
// chunks permuted by swz_col.
template <bool SWZ = false, class Epi>
__device__ __forceinline__ void gemm_hl(const HL& A, int n, int K, const __nv_bfloat16* Wt,
                                        int ldw, int Os, Epi epi) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int mi = lane >> 3, rr = lane & 7;
  const int mt = (n + 15) >> 4, np = Os >> 3;
  const int kr = lane & 15;  // B row of this lane within a 16-row k step (lanes 16..31 unused)
#pragma unroll 1
  for (int unit = warp; unit < mt * np; unit += (blockDim.x >> 5)) {
    const int m0 = (unit / np) * 16, c0 = (unit % np) * 8;
    float acc[4] = {0.f, 0.f, 0.f, 0.f}, acl[4] = {0.f, 0.f, 0.f, 0.f};
    const uint32_t ah_base =
        smem_u32(A.p + (m0 + (mi & 1) * 8 + rr) * A.ld + (mi >> 1) * 8);
    const uint32_t al_base = ah_base + static_cast<uint32_t>(A.plane * 2);
    const int ch = c0 >> 3;
    const uint32_t w_base =
        smem_u32(Wt + kr * ldw + 8 * (SWZ ? (ch ^ rimg::swz_mask(kr, ldw)) : ch));
#pragma unroll 2
    for (int k0 = 0; k0 < K; k0 += 16) {
      uint32_t ah[4], al[4], b0, b1;
      ldsm_x4(ah_base + k0 * 2, ah[0], ah[1], ah[2], ah[3]);
      ldsm_x4(al_base + k0 * 2, al[0], al[1], al[2], al[3]);
      ldsm_x2_t(w_base + static_cast<uint32_t>(k0 * ldw * 2), b0, b1);
      mma_bf16(acc, ah, b0, b1);
      mma_bf16(acl, al, b0, b1);
    }
    const int r_lo = m0 + g, r_hi = r_lo + 8;
    const int o = c0 + 2 * t;
    if (r_lo < n) epi(r_lo, o, acc[0] + acl[0], acc[1] + acl[1]);
    if (r_hi < n) epi(r_hi, o, acc[2] + acl[2], acc[3] + acl[3]);
  }
}

// Sum over the 8 lanes of an aligned lane group.
__device__ __forceinline__ float group8_sum(float v) {
  v += __shfl_xor_sync(0xffffffffu, v, 1);
  v += __shfl_xor_sync(0xffffffffu, v, 2);
  v += __shfl_xor_sync(0xffffffffu, v, 4);
  return v;
}

// LayerNorm (eps 1e-5) over DIM (32, 64 or 128) features of rows j < n:
// 8 lanes per row, lane q holding columns 4q + 32c (c < DIM/32); the result
// goes to the hi/lo buffer hl and, if DST, to an fp32 buffer (which may be
// src itself: every lane reads its values before it writes them).
template <int DIM, bool DST>
__device__ __forceinline__ void ln_rows(const float* src, int lds, float* dst, int ldd, const HL hl,
                                        int n, const float* g, const float* b) {
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
        const float4 bb = *reinterpret_cast<const float4*>(b + o);
        const float4 y = make_float4((v[c].x - mean) * inv * gg.x + bb.x, (v[c].y - mean) * inv * gg.y + bb.y,
                                     (v[c].z - mean) * inv * gg.z + bb.z, (v[c].w - mean) * inv * gg.w + bb.w);
        if (DST) *reinterpret_cast<float4*>(dst + j * ldd + o) = y;
        uint32_t h0, l0, h1, l1;
        split_bf16x2(y.x, y.y, h0, l0);
        split_bf16x2(y.z, y.w, h1, l1);
        *reinterpret_cast<uint2*>(hl.p + j * hl.ld + o) = make_uint2(h0, h1);
        *reinterpret_cast<uint2*>(hl.p + hl.plane + j * hl.ld + o) = make_uint2(l0, l1);
      }
    }
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

// ------------------------------------------------------------------ LPS
// One attention unit: 16 query rows [m0, m0+16) of head h (width 8) over the
// n keys, in blocks of 16 keys with a running max and sum (the result is
// softmax(q k^T / sqrt(8)) v, the blocks only bound the live registers);
// qkv: [n][100] fp32 (q | k | v); the output goes to hi/lo columns
// 8h..8h+7 of `out`.
__device__ __forceinline__ void lps_attention_unit(const float* qkv, int n, int m0, int h,
                                                   const HL& out) {
  const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const int r_lo = m0 + g, r_hi = r_lo + 8;
  uint32_t qh[4], ql[4];
  {
    float2 q0 = make_float2(0.f, 0.f), q1 = make_float2(0.f, 0.f);
    if (r_lo < n) q0 = *reinterpret_cast<const float2*>(qkv + r_lo * 100 + 8 * h + 2 * t);
    if (r_hi < n) q1 = *reinterpret_cast<const float2*>(qkv + r_hi * 100 + 8 * h + 2 * t);
    split_bf16x2(q0.x, q0.y, qh[0], ql[0]);
    split_bf16x2(q1.x, q1.y, qh[1], ql[1]);
    qh[2] = qh[3] = ql[2] = ql[3] = 0u;  // head width 8: upper k half is zero
  }
  const float scale = 0.35355339059327373f;  // 1/sqrt(8)
  float mx0 = -INFINITY, mx1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float o[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
  for (int k0 = 0; k0 < n; k0 += 16) {
    float s[2][4];
#pragma unroll
    for (int hb = 0; hb < 2; ++hb) {
      const int key = k0 + 8 * hb + g;
      const float2 kk = key < n ? *reinterpret_cast<const float2*>(qkv + key * 100 + 32 + 8 * h + 2 * t)
                                : make_float2(0.f, 0.f);
      uint32_t bh, bl;
      split_bf16x2(kk.x, kk.y, bh, bl);
      float a[4] = {0.f, 0.f, 0.f, 0.f};
      mma_bf16(a, qh, bh, 0u);
      mma_bf16(a, qh, bl, 0u);
      mma_bf16(a, ql, bh, 0u);
      const int c = k0 + 8 * hb + 2 * t;
      s[hb][0] = c < n ? a[0] * scale : -INFINITY;
      s[hb][1] = c + 1 < n ? a[1] * scale : -INFINITY;
      s[hb][2] = c < n ? a[2] * scale : -INFINITY;
      s[hb][3] = c + 1 < n ? a[3] * scale : -INFINITY;
    }
    float b0 = fmaxf(fmaxf(s[0][0], s[0][1]), fmaxf(s[1][0], s[1][1]));
    float b1 = fmaxf(fmaxf(s[0][2], s[0][3]), fmaxf(s[1][2], s[1][3]));
    b0 = fmaxf(b0, __shfl_xor_sync(0xffffffffu, b0, 1));
    b0 = fmaxf(b0, __shfl_xor_sync(0xffffffffu, b0, 2));
    b1 = fmaxf(b1, __shfl_xor_sync(0xffffffffu, b1, 1));
    b1 = fmaxf(b1, __shfl_xor_sync(0xffffffffu, b1, 2));
    const float n0 = fmaxf(mx0, b0), n1 = fmaxf(mx1, b1);  // finite: key k0 is valid
    const float c0 = expf(mx0 - n0), c1 = expf(mx1 - n1);
    mx0 = n0;
    mx1 = n1;
#pragma unroll
    for (int hb = 0; hb < 2; ++hb) {
      s[hb][0] = expf(s[hb][0] - n0);
      s[hb][1] = expf(s[hb][1] - n0);
      s[hb][2] = expf(s[hb][2] - n1);
      s[hb][3] = expf(s[hb][3] - n1);
    }
    l0 = l0 * c0 + ((s[0][0] + s[0][1]) + (s[1][0] + s[1][1]));
    l1 = l1 * c1 + ((s[0][2] + s[0][3]) + (s[1][2] + s[1][3]));
    o[0] *= c0;
    o[1] *= c0;
    o[2] *= c1;
    o[3] *= c1;
    uint32_t ph[4], pl[4];
    split_bf16x2(s[0][0], s[0][1], ph[0], pl[0]);
    split_bf16x2(s[0][2], s[0][3], ph[1], pl[1]);
    split_bf16x2(s[1][0], s[1][1], ph[2], pl[2]);
    split_bf16x2(s[1][2], s[1][3], ph[3], pl[3]);
    float v[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int key = k0 + (e >> 1) * 8 + 2 * t + (e & 1);
      v[e] = key < n ? qkv[key * 100 + 64 + 8 * h + g] : 0.f;
    }
    uint32_t v0h, v0l, v1h, v1l;
    split_bf16x2(v[0], v[1], v0h, v0l);
    split_bf16x2(v[2], v[3], v1h, v1l);
    mma_bf16(o, ph, v0h, v1h);
    mma_bf16(o, ph, v0l, v1l);
    mma_bf16(o, pl, v0h, v1h);
  }
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float i0 = 1.0f / l0, i1 = 1.0f / l1;
  if (r_lo < n) hl_store2(out, r_lo, 8 * h + 2 * t, o[0] * i0, o[1] * i0);
  if (r_hi < n) hl_store2(out, r_hi, 8 * h + 2 * t, o[2] * i1, o[3] * i1);
}

// LPS (Sec. 5.2 / App. D.1): Linear(5->32) -> LayerNorm -> GELU, two pre-norm
// blocks (4 heads of width 8, FFN 64, GELU), head Linear(32->1), p = sigmoid.
// Over the n (<= 64) masked rows of the block (features at P + L_FEAT);
// p_psi of row i -> P[L_PROB + i].  Called by the whole CTA.  Phases: 0 the
// input layer; per block 1 LN1, 2 QKV, 3 attention, 4 output projection,
// 5 LN2, 6 FF1, 7 FF2; 8 the second block and the head.  Only phases
// [from, to] of the first block run (from = 8: none of it); the second
// block and the head run when to = 8.  Only the stand-in runs of the
// decision kernel pass anything but [0, 8].
__device__ __noinline__ void lps_forward(float* P, int n, const __nv_bfloat16* Wlps,
                                         const float* V, int from, int to) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float* feats = P + L_FEAT;
  float* Z = P + L_Z;
  float* QKV = P + L_QKV;
  const HL Y = hl_at(P + L_YH, 40);
  const HL At = hl_at(P + L_AH, 40);
  const HL Hh = hl_at(P + L_HH, 72);
  if (from <= 0 && to >= 0) {  // Linear(5 -> 32), LayerNorm, GELU: 8 lanes per row, 4 outputs each
    const int q = lane & 7;
#pragma unroll 1
    for (int j0 = 0; j0 < n; j0 += (blockDim.x >> 3)) {
      const int j = j0 + (tid >> 3);
      const bool ok = j < n;
      float y[4];
      float s = 0.f;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int c = 4 * q + e;
        float a = V[VP_INB + c];
#pragma unroll
        for (int k = 0; k < 5; ++k) a = fmaf(ok ? feats[j * 8 + k] : 0.f, V[VP_INT + k * 32 + c], a);
        y[e] = a;
        s += a;
      }
      const float mean = group8_sum(s) * (1.0f / 32.0f);
      float var = 0.f;
#pragma unroll
      for (int e = 0; e < 4; ++e) var += (y[e] - mean) * (y[e] - mean);
      const float inv = 1.0f / sqrtf(group8_sum(var) * (1.0f / 32.0f) + 1e-5f);
      if (ok) {
        float4 z;
        z.x = gelu((y[0] - mean) * inv * V[VP_INLNG + 4 * q + 0] + V[VP_INLNB + 4 * q + 0]);
        z.y = gelu((y[1] - mean) * inv * V[VP_INLNG + 4 * q + 1] + V[VP_INLNB + 4 * q + 1]);
        z.z = gelu((y[2] - mean) * inv * V[VP_INLNG + 4 * q + 2] + V[VP_INLNB + 4 * q + 2]);
        z.w = gelu((y[3] - mean) * inv * V[VP_INLNG + 4 * q + 3] + V[VP_INLNB + 4 * q + 3]);
        *reinterpret_cast<float4*>(Z + j * LDQ + 4 * q) = z;
      }
    }
  }
  __syncthreads();
#pragma unroll 1
  for (int l = 0; l < 2; ++l) {
    if (l == 1 && to < 8) break;
    const __nv_bfloat16* Wl = Wlps + l * PL_STRIDE;
    const float* Vl = V + VP_LAYER0 + l * VP_LAYER_STRIDE;
    const int f = l == 0 ? from : 0, t = l == 0 ? to : 8;
    if (f <= 1 && t >= 1) ln_rows<32, false>(Z, LDQ, nullptr, 0, Y, n, Vl + VPL_LN1G, Vl + VPL_LN1B);
    __syncthreads();
    if (f <= 2 && t >= 2)
      gemm_hl(Y, n, 32, Wl + PL_QKV, PL_LDQKV, 96, [&](int j, int o, float a, float b) {
        *reinterpret_cast<float2*>(QKV + j * 100 + o) = make_float2(a + Vl[VPL_QKVB + o], b + Vl[VPL_QKVB + o + 1]);
      });
    __syncthreads();
    const int mt = (n + 15) >> 4;
    if (f <= 3 && t >= 3) {
#pragma unroll 1
      for (int u = warp; u < 4 * mt; u += (blockDim.x >> 5)) lps_attention_unit(QKV, n, 16 * (u >> 2), u & 3, At);
    }
    __syncthreads();
    if (f <= 4 && t >= 4)
      gemm_hl(At, n, 32, Wl + PL_OUT, PL_LDOUT, 32, [&](int j, int o, float a, float b) {
        float2* z = reinterpret_cast<float2*>(Z + j * LDQ + o);
        const float2 zz = *z;
        *z = make_float2(zz.x + (a + Vl[VPL_OUTB + o]), zz.y + (b + Vl[VPL_OUTB + o + 1]));
      });
    __syncthreads();
    if (f <= 5 && t >= 5) ln_rows<32, false>(Z, LDQ, nullptr, 0, Y, n, Vl + VPL_LN2G, Vl + VPL_LN2B);
    __syncthreads();
    if (f <= 6 && t >= 6)
      gemm_hl(Y, n, 32, Wl + PL_FF1, PL_LDFF1, 64, [&](int j, int o, float a, float b) {
        hl_store2(Hh, j, o, gelu(a + Vl[VPL_FF1B + o]), gelu(b + Vl[VPL_FF1B + o + 1]));
      });
    __syncthreads();
    if (f <= 7 && t >= 7)
      gemm_hl(Hh, n, 64, Wl + PL_FF2, PL_LDFF2, 32, [&](int j, int o, float a, float b) {
        float2* z = reinterpret_cast<float2*>(Z + j * LDQ + o);
        const float2 zz = *z;
        *z = make_float2(zz.x + (a + Vl[VPL_FF2B + o]), zz.y + (b + Vl[VPL_FF2B + o + 1]));
      });
    __syncthreads();
  }
  if (to < 8) return;
#pragma unroll 1
  for (int i = warp; i < n; i += (blockDim.x >> 5)) {
    const float a = warp_sum(Z[i * LDQ + lane] * V[VP_HEADW + lane]) + V[VP_HEADB];
    if (lane == 0) P[L_PROB + i] = 1.0f / (1.0f + expf(-a));
  }
  __syncthreads();
}

}  // namespace
}  // namespace ebd
