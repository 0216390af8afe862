// Window attention: the active window's queries attend, without a mask, to
// the sequence's cached prefix keys, the window's own keys and, with a dual
// cache, a cached suffix range (bidirectional dLLM, Sec. 3; prefix and dual
// cache at the block boundaries, Sec. 6.3).
//   O = softmax(Q K^T / sqrt(D)) V, fp32 output.
// The key range is a list of 64-key chunks: prefix tiles of the cache, one
// tile of window rows, then suffix tiles of the cache.  Both kernels below
// take a query tile of 64 rows (query head of the kv group, window row) and
// one split of the chunks per CTA, grid (key split, query tile, sequence x
// kv head); splits of the key range combine their (max, sum, O) partials in
// the last CTA to finish (atomic ticket).  K/V tiles are staged by TMA with
// a 128-byte swizzle.  The probabilities are split into a bf16 high part and
// a bf16 remainder, so that P V keeps ~16 mantissa bits.
//   attn_tc_kernel: the 5th-generation tensor cores (S and O in TMEM); one
//     CTA per SM; for long key ranges and launches of few tiles.
//   attn_kernel: mma.sync, 4 warps of 16 query rows, a 3-stage K/V ring, two
//     CTAs per SM; for launches of many tiles with short key ranges, where
//     the tcgen05 kernel's per-CTA setup does not amortise.
#include <type_traits>

#include "internal.h"
#include "ptx.cuh"

namespace ebd {

namespace {

constexpr int kStageBytes = 4 * 8192;  // K and V, two 64-dim halves each

// byte offset of 16-byte chunk `c` (0..7) of row `r` in a 128B-swizzled tile
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return static_cast<uint32_t>(r * 128 + ((c ^ (r & 7)) << 4));
}

// ---------------------------------------------------------------- tcgen05 kernel
// Shared-memory map of the tcgen05 attention CTA (offsets from a 1024-byte
// aligned base).  A step covers 128 keys (two 64-key chunks):
//   Q    [NB boxes][128 rows][128 B]  (64 query rows, repeated)
//   K, V rings of kTcRing steps, each [NB boxes][128 keys][128 B]
//   P    [2 key blocks of 64][128 rows][128 B]: bf16 high parts in rows
//        0..63, low parts in rows 64..127
//   barriers, then the row maxima / sums exchanged between the warps that
//   share a query row.
constexpr int kTcRing = 2;
constexpr int kTcKeys = 128;  // keys per step
template <int D>
struct TcMap {
  static constexpr int NB = D / 64;                          // 64-dim boxes
  static constexpr uint32_t kBox = 8192;                     // 64 keys x 64 dims
  static constexpr uint32_t kStep = NB * 2 * kBox;           // one ring slot: 128 keys
  static constexpr uint32_t kQ = 0;
  static constexpr uint32_t kK0 = NB * 16384;
  static constexpr uint32_t kV0 = kK0 + kTcRing * kStep;
  static constexpr uint32_t kP0 = kV0 + kTcRing * kStep;
  static constexpr uint32_t kBar = kP0 + 32768;
  static constexpr int kNBar = 4 * kTcRing + 8;              // k/v full and empty, s_full[2],
                                                             // s_free[2], p_full, pv_done, drain,
                                                             // q_ready
  static constexpr uint32_t kXm = kBar + kNBar * 8;          // float [2][8][64]
  static constexpr uint32_t kXl = kXm + 2 * 8 * 64 * 4;      // float [8][64]
  static constexpr uint32_t kMisc = kXl + 8 * 64 * 4;        // TMEM base, abort flag, ticket flag
  static constexpr uint32_t kBytes = kMisc + 16;
  // at least half of the SM's shared memory: one CTA per SM, whose 512 TMEM
  // columns it then holds alone
  static constexpr uint32_t kDyn = (kBytes + 1024) > 120u * 1024 ? kBytes + 1024 : 120u * 1024;
};
constexpr uint32_t kTcTmemCols = 512;  // S double buffer (2 x 128) + O (up to 128)

// Shared-memory descriptor of an MN-major operand with 128-byte swizzle:
// 64 contiguous elements along MN per 128-byte row, rows along K, 8-row
// groups 1024 bytes apart (stride byte offset), 64-element MN blocks `lbo`
// bytes apart (leading byte offset).
__device__ __forceinline__ uint64_t umma_desc_mn_sw128(uint32_t smem_addr, uint32_t lbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((smem_addr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>(1024u >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 32 lanes x N consecutive 32-bit columns (N = 8, 16, 32) into registers
template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, float (&v)[N]);
template <>
__device__ __forceinline__ void tmem_ld_cols<8>(uint32_t taddr, float (&v)[8]) {
  uint32_t r[8];
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
                 "=r"(r[6]), "=r"(r[7])
               : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}
template <>
__device__ __forceinline__ void tmem_ld_cols<16>(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
template <>
__device__ __forceinline__ void tmem_ld_cols<32>(uint32_t taddr, float (&v)[32]) {
  tmem_ld_32x32b_x32(taddr, v);
}

// 32 lanes x 32 consecutive 32-bit columns from registers (lane = thread)
__device__ __forceinline__ void tmem_st_32x32b_x32(uint32_t taddr, const float (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

}  // namespace

template <int D>
__device__ __forceinline__ void attn_body(const CUtensorMap& tm_kc, const CUtensorMap& tm_vc,
                                          const CUtensorMap& tm_kw, const CUtensorMap& tm_vw,
                                          const AttnParams& p) {
  constexpr int NH = D / 64;   // 64-dim halves
  constexpr int KS = D / 16;   // k-steps of Q K^T
  constexpr int NT = D / 8;    // n-tiles of the output
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kAttnStages * kStageBytes);
  __shared__ int s_flag;

  const int split = blockIdx.x, qt = blockIdx.y, bg = blockIdx.z;
  const int b = bg / p.Hkv, g = bg - b * p.Hkv;
  const int r0 = p.cu_rows[b];
  const int wb = p.cu_rows[b + 1] - r0;
  const int m_total = wb * p.group;
  if (wb <= 0 || wb > kMaxWindow || qt * 64 >= m_total) return;
  if (!in_bounds(r0, p.R, p.status) || !in_bounds(r0 + wb - 1, p.R, p.status)) return;
  int P = p.prefix_len[b];
  P = P < 0 ? 0 : (P > p.max_prefix ? p.max_prefix : P);
  int S0 = 0, S = 0;  // suffix range of the cache (dual cache)
  if (p.suffix != nullptr) {
    S0 = min(max(p.suffix[2 * b], 0), p.max_prefix);
    S = min(max(p.suffix[2 * b + 1], 0), p.max_prefix - S0);
  }
  const int ncc = (P + kAttnChunk - 1) / kAttnChunk;
  const int nch = ncc + 1 + (S + kAttnChunk - 1) / kAttnChunk;
  const int c0 = static_cast<int>((static_cast<long long>(split) * nch) / p.splits);
  const int c1 = static_cast<int>((static_cast<long long>(split + 1) * nch) / p.splits);
  const int nmy = c1 - c0;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int s = 0; s < kAttnStages; ++s) mbar_init(&full[s], 1);
    fence_mbar_init();
    s_flag = 0;
  }
  __syncthreads();

  auto issue = [&](int i) {
    const int s = i % kAttnStages;
    const int c = c0 + i;
    uint8_t* kd = smem + s * kStageBytes;
    uint8_t* vd = kd + 2 * 8192;
    mbar_arrive_expect_tx(&full[s], 2u * NH * 8192u);
#pragma unroll
    for (int hf = 0; hf < NH; ++hf) {
      if (c < ncc) {
        tma_load_4d(kd + hf * 8192, &tm_kc, &full[s], hf * 64, g, c * kAttnChunk, b);
        tma_load_4d(vd + hf * 8192, &tm_vc, &full[s], hf * 64, g, c * kAttnChunk, b);
      } else if (c == ncc) {
        tma_load_3d(kd + hf * 8192, &tm_kw, &full[s], hf * 64, g, r0);
        tma_load_3d(vd + hf * 8192, &tm_vw, &full[s], hf * 64, g, r0);
      } else {
        const int y = S0 + (c - ncc - 1) * kAttnChunk;
        tma_load_4d(kd + hf * 8192, &tm_kc, &full[s], hf * 64, g, y, b);
        tma_load_4d(vd + hf * 8192, &tm_vc, &full[s], hf * 64, g, y, b);
      }
    }
  };
  if (tid == 0)
    for (int i = 0; i < nmy && i < kAttnStages; ++i) issue(i);

  // query fragments of this warp's 16 rows
  const int mrow_lo = qt * 64 + warp * 16 + (lane >> 2);
  const int mrow_hi = mrow_lo + 8;
  auto qptr = [&](int m) -> const __nv_bfloat16* {
    if (m >= m_total) return nullptr;
    const int hl = m / wb, r = m - hl * wb;
    return p.q + (static_cast<size_t>(r0 + r) * p.Hq + g * p.group + hl) * D;
  };
  const __nv_bfloat16* q_lo = qptr(mrow_lo);
  const __nv_bfloat16* q_hi = qptr(mrow_hi);
  const bool warp_active = qt * 64 + warp * 16 < m_total;
  uint32_t qf[KS][4];
#pragma unroll
  for (int ks = 0; ks < KS; ++ks) {
    const int c = ks * 16 + 2 * (lane & 3);
    qf[ks][0] = q_lo ? *reinterpret_cast<const uint32_t*>(q_lo + c) : 0u;
    qf[ks][1] = q_hi ? *reinterpret_cast<const uint32_t*>(q_hi + c) : 0u;
    qf[ks][2] = q_lo ? *reinterpret_cast<const uint32_t*>(q_lo + c + 8) : 0u;
    qf[ks][3] = q_hi ? *reinterpret_cast<const uint32_t*>(q_hi + c + 8) : 0u;
  }

  float o[NT][4];
#pragma unroll
  for (int t = 0; t < NT; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;
  float m_lo = -INFINITY, m_hi = -INFINITY, l_lo = 0.f, l_hi = 0.f;
  const float sl2 = 1.4426950408889634f / sqrtf(static_cast<float>(D));  // log2(e)/sqrt(D)

  bool failed = false;
  for (int i = 0; i < nmy; ++i) {
    const int s = i % kAttnStages;
    const bool ok = mbar_wait(&full[s], static_cast<uint32_t>(i / kAttnStages) & 1u, p.limit_ns,
                              nullptr);
    if (__syncthreads_or(!ok)) {
      failed = true;
      if (tid == 0) {
        atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
        for (int j = i; j < nmy && j < i + kAttnStages; ++j)
          mbar_wait(&full[j % kAttnStages], static_cast<uint32_t>(j / kAttnStages) & 1u,
                    p.limit_ns, nullptr);
      }
      break;
    }
    const int c = c0 + i;
    const int nvalid = c < ncc ? min(kAttnChunk, P - c * kAttnChunk)
                       : (c == ncc ? wb : min(kAttnChunk, S - (c - ncc - 1) * kAttnChunk));
    const uint32_t kbase = smem_u32(smem + s * kStageBytes);
    const uint32_t vbase = kbase + 2 * 8192;
    if (warp_active) {
      float sc[8][4];
#pragma unroll
      for (int t = 0; t < 8; ++t) sc[t][0] = sc[t][1] = sc[t][2] = sc[t][3] = 0.f;
      const int mi = lane >> 3, rr = lane & 7;
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        const int hf = ks >> 2;
        const int cidx = (ks & 3) * 2;
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          const int key = np * 16 + (mi >> 1) * 8 + rr;
          const uint32_t addr = kbase + hf * 8192 + swz(key, cidx + (mi & 1));
          uint32_t b0, b1, b2, b3;
          ldsm_x4(addr, b0, b1, b2, b3);
          mma_bf16(sc[2 * np], qf[ks], b0, b1);
          mma_bf16(sc[2 * np + 1], qf[ks], b2, b3);
        }
      }
      float mx_lo = -INFINITY, mx_hi = -INFINITY;
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const int k0 = t * 8 + 2 * (lane & 3);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = k0 + (e & 1);
          const float v = key < nvalid ? sc[t][e] * sl2 : -INFINITY;
          sc[t][e] = v;
        }
        mx_lo = fmaxf(mx_lo, fmaxf(sc[t][0], sc[t][1]));
        mx_hi = fmaxf(mx_hi, fmaxf(sc[t][2], sc[t][3]));
      }
#pragma unroll
      for (int off = 1; off <= 2; off <<= 1) {
        mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, off));
        mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, off));
      }
      const float mn_lo = fmaxf(m_lo, mx_lo), mn_hi = fmaxf(m_hi, mx_hi);
      const float al_lo = exp2f(m_lo - mn_lo), al_hi = exp2f(m_hi - mn_hi);
      m_lo = mn_lo;
      m_hi = mn_hi;
      float sum_lo = 0.f, sum_hi = 0.f;
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        sc[t][0] = exp2f(sc[t][0] - mn_lo);
        sc[t][1] = exp2f(sc[t][1] - mn_lo);
        sc[t][2] = exp2f(sc[t][2] - mn_hi);
        sc[t][3] = exp2f(sc[t][3] - mn_hi);
        sum_lo += sc[t][0] + sc[t][1];
        sum_hi += sc[t][2] + sc[t][3];
      }
#pragma unroll
      for (int off = 1; off <= 2; off <<= 1) {
        sum_lo += __shfl_xor_sync(0xffffffffu, sum_lo, off);
        sum_hi += __shfl_xor_sync(0xffffffffu, sum_hi, off);
      }
      l_lo = l_lo * al_lo + sum_lo;
      l_hi = l_hi * al_hi + sum_hi;
#pragma unroll
      for (int t = 0; t < NT; ++t) {
        o[t][0] *= al_lo;
        o[t][1] *= al_lo;
        o[t][2] *= al_hi;
        o[t][3] *= al_hi;
      }
      // O += P V, P split into bf16 high and low parts
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t ah[4], al[4];
        split_bf16x2(sc[2 * kk][0], sc[2 * kk][1], ah[0], al[0]);
        split_bf16x2(sc[2 * kk][2], sc[2 * kk][3], ah[1], al[1]);
        split_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1], ah[2], al[2]);
        split_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3], ah[3], al[3]);
#pragma unroll
        for (int dp = 0; dp < D / 16; ++dp) {
          const int hf = dp >> 2;
          const int key = kk * 16 + (mi & 1) * 8 + rr;
          const int chunk = (dp & 3) * 2 + (mi >> 1);
          const uint32_t addr = vbase + hf * 8192 + swz(key, chunk);
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(addr, b0, b1, b2, b3);
          mma_bf16(o[2 * dp], ah, b0, b1);
          mma_bf16(o[2 * dp], al, b0, b1);
          mma_bf16(o[2 * dp + 1], ah, b2, b3);
          mma_bf16(o[2 * dp + 1], al, b2, b3);
        }
      }
    }
    __syncthreads();
    if (tid == 0 && i + kAttnStages < nmy) issue(i + kAttnStages);
  }
  if (failed) return;

  // ------------------------------------------------------------ output / partials
  auto out_row = [&](int m) -> float* {
    const int hl = m / wb, r = m - hl * wb;
    return p.out + (static_cast<size_t>(r0 + r) * p.Hq + g * p.group + hl) * D;
  };
  if (p.splits == 1) {
    if (warp_active) {
      const float il = l_lo > 0.f ? 1.0f / l_lo : 0.f, ih = l_hi > 0.f ? 1.0f / l_hi : 0.f;
#pragma unroll
      for (int t = 0; t < NT; ++t) {
        const int d = t * 8 + 2 * (lane & 3);
        if (mrow_lo < m_total && in_bounds(r0 + mrow_lo % wb, p.R, p.status))
          *reinterpret_cast<float2*>(out_row(mrow_lo) + d) = make_float2(o[t][0] * il, o[t][1] * il);
        if (mrow_hi < m_total && in_bounds(r0 + mrow_hi % wb, p.R, p.status))
          *reinterpret_cast<float2*>(out_row(mrow_hi) + d) = make_float2(o[t][2] * ih, o[t][3] * ih);
      }
    }
    return;
  }
  const int slot = (bg * p.max_qtiles + qt);
  // partials: O rows [slot][split][64][D] and (max, sum) [slot][split][64][2]
  float* po = p.part + (static_cast<size_t>(slot) * p.splits + split) * 64 * D;
  float* pml = p.part_ml + (static_cast<size_t>(slot) * p.splits + split) * 64 * 2;
  if (warp_active) {
    const int ml = warp * 16 + (lane >> 2), mh = ml + 8;
#pragma unroll
    for (int t = 0; t < NT; ++t) {
      const int d = t * 8 + 2 * (lane & 3);
      *reinterpret_cast<float2*>(po + ml * D + d) = make_float2(o[t][0], o[t][1]);
      *reinterpret_cast<float2*>(po + mh * D + d) = make_float2(o[t][2], o[t][3]);
    }
    if ((lane & 3) == 0) {
      *reinterpret_cast<float2*>(pml + ml * 2) = make_float2(m_lo, l_lo);
      *reinterpret_cast<float2*>(pml + mh * 2) = make_float2(m_hi, l_hi);
    }
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) s_flag = (atomicAdd(&p.tickets[slot], 1) == p.splits - 1);
  __syncthreads();
  if (!s_flag) return;
  __threadfence();
  // last CTA of the slot: per-row split weights, then a weighted sum of the
  // splits' O rows with independent vector loads
  __shared__ float s_w[64][kMaxAttnSplits];
  const float* bo = p.part + static_cast<size_t>(slot) * p.splits * 64 * D;
  const float* bml = p.part_ml + static_cast<size_t>(slot) * p.splits * 64 * 2;
  const int rows_here = min(64, m_total - qt * 64);
  for (int r = tid; r < rows_here; r += blockDim.x) {
    float M = -INFINITY;
    for (int sp = 0; sp < p.splits; ++sp) M = fmaxf(M, bml[(sp * 64 + r) * 2]);
    float L = 0.f;
    for (int sp = 0; sp < p.splits; ++sp) {
      const float2 v = *reinterpret_cast<const float2*>(bml + (sp * 64 + r) * 2);
      const float wgt = v.x == -INFINITY ? 0.f : exp2f(v.x - M);
      s_w[r][sp] = wgt;
      L += wgt * v.y;
    }
    const float inv = L > 0.f ? 1.0f / L : 0.f;
    for (int sp = 0; sp < p.splits; ++sp) s_w[r][sp] *= inv;
  }
  __syncthreads();
  constexpr int D4 = D / 4;
  for (int it = tid; it < rows_here * D4; it += blockDim.x) {
    const int r = it / D4, d = (it - r * D4) * 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int sp = 0; sp < kMaxAttnSplits; ++sp) {
      if (sp < p.splits) {
        const float4 v = __ldcg(reinterpret_cast<const float4*>(bo + (static_cast<size_t>(sp) * 64 + r) * D + d));
        const float wgt = s_w[r][sp];
        acc.x = fmaf(wgt, v.x, acc.x);
        acc.y = fmaf(wgt, v.y, acc.y);
        acc.z = fmaf(wgt, v.z, acc.z);
        acc.w = fmaf(wgt, v.w, acc.w);
      }
    }
    if (in_bounds(r0 + (qt * 64 + r) % wb, p.R, p.status))
      *reinterpret_cast<float4*>(out_row(qt * 64 + r) + d) = acc;
  }
  if (tid == 0) p.tickets[slot] = 0;
}

__device__ __forceinline__ bool named_barrier_and(uint32_t id, uint32_t n, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred q, %2, %3, p;\n"
      " selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(id), "r"(n)
      : "memory");
  return r != 0;
}

// The same attention on the 5th-generation tensor cores.  A CTA takes 64
// query rows of one (sequence, kv head) -- rows past the group's window
// rows are zero -- and one split of the key chunks, in steps of 128 keys.
//   warps 0 and 10: TMA loads of the K steps and of the V steps, each into
//           its own ring of 2 steps (a K slot frees after its Q K^T, a V slot
//           after its P V);
//   warp 1: TMEM allocation and the MMA thread: S = Q K^T (M = 128, N = 128,
//           both operands K-major) into one of two 128-column TMEM buffers,
//           then O += P V with M = 128: rows 0..63 of P hold the
//           probabilities' bf16 high parts and rows 64..127 their low parts
//           (~16 mantissa bits in all), so TMEM lanes r and 64 + r accumulate
//           the two halves of query row r's output; V is an MN-major operand
//           (head dims contiguous, as TMA stored the tile);
//   warps 2-9: the softmax.  The query tile repeats its rows over the four
//           TMEM lane quadrants (32 rows: four copies; 64 rows: two), and
//           each warp reads its own quadrant (only the warps of one SM
//           sub-partition can) for a share of every step's keys: 16 of 128
//           (32 rows) or 32 (64 rows).  The warps sharing a query row
//           exchange their maxima and sums through shared memory.
// The running maximum m moves only when a step's maximum exceeds it by more
// than 8 (log2 units), so that every exp2(s - m) stays below 256; O is then
// rescaled in TMEM, after the previous P V has completed.
template <int D>
__device__ __forceinline__ void attn_tc_body(const CUtensorMap& tm_kc, const CUtensorMap& tm_vc,
                                             const CUtensorMap& tm_kw, const CUtensorMap& tm_vw,
                                             const AttnParams& p) {
  using L = TcMap<D>;
  constexpr int NB = L::NB;
  constexpr int HALF = D / 2;  // O columns per warp
  constexpr int TR = kAttnTcRows;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::kBar);
  uint64_t* kfull = bars;
  uint64_t* kempty = kfull + kTcRing;
  uint64_t* vfull = kempty + kTcRing;
  uint64_t* vempty = vfull + kTcRing;
  uint64_t* s_full = vempty + kTcRing;
  uint64_t* s_free = s_full + 2;
  uint64_t* p_full = s_free + 2;
  uint64_t* pv_done = p_full + 1;
  uint64_t* drain = pv_done + 1;
  uint64_t* q_ready = drain + 1;
  float* xm = reinterpret_cast<float*>(smem + L::kXm);
  float* xl = reinterpret_cast<float*>(smem + L::kXl);
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(smem + L::kMisc);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + L::kMisc + 4);
  int* s_flag = reinterpret_cast<int*>(smem + L::kMisc + 8);

  const int split = blockIdx.x, qt = blockIdx.y, bg = blockIdx.z;
  const int b = bg / p.Hkv, g = bg - b * p.Hkv;
  const int r0 = p.cu_rows[b];
  const int wb = p.cu_rows[b + 1] - r0;
  const int m_total = wb * p.group;
  if (wb <= 0 || wb > kMaxWindow || qt * TR >= m_total) return;
  if (!in_bounds(r0, p.R, p.status) || !in_bounds(r0 + wb - 1, p.R, p.status)) return;
  int P = p.prefix_len[b];
  P = P < 0 ? 0 : (P > p.max_prefix ? p.max_prefix : P);
  int S0 = 0, S = 0;  // suffix range of the cache (dual cache)
  if (p.suffix != nullptr) {
    S0 = min(max(p.suffix[2 * b], 0), p.max_prefix);
    S = min(max(p.suffix[2 * b + 1], 0), p.max_prefix - S0);
  }
  const int ncc = (P + kAttnChunk - 1) / kAttnChunk;
  const int nch = ncc + 1 + (S + kAttnChunk - 1) / kAttnChunk;
  const int c0 = static_cast<int>((static_cast<long long>(split) * nch) / p.splits);
  const int c1 = static_cast<int>((static_cast<long long>(split + 1) * nch) / p.splits);
  const int nmy = c1 - c0;              // 64-key chunks of this split
  const int nst = (nmy + 1) / 2;        // steps of two chunks
  const int slot = bg * p.max_qtiles + qt;
  const int m_tile = m_total - qt * TR;
  const int nrow = m_tile <= 32 ? 32 : 64;  // distinct query rows held per 128 tile rows
  auto nvalid = [&](int k) {  // valid keys of chunk k of this split (0 past its end)
    if (k >= nmy) return 0;
    const int c = c0 + k;
    return c < ncc ? min(kAttnChunk, P - c * kAttnChunk)
                   : (c == ncc ? wb : min(kAttnChunk, S - (c - ncc - 1) * kAttnChunk));
  };

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int s = 0; s < kTcRing; ++s) {
      mbar_init(&kfull[s], 1);
      mbar_init(&kempty[s], 1);
      mbar_init(&vfull[s], 1);
      mbar_init(&vempty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 8);  // one arrival per softmax warp
    }
    mbar_init(p_full, 8);
    mbar_init(pv_done, 1);
    mbar_init(drain, 1);
    mbar_init(q_ready, 9);  // warps 1..9 fill the query tile
    *abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_holder, kTcTmemCols);
  tc_fence_before();
  __syncthreads();  // barriers initialised, TMEM allocated
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  if (warp >= 1 && warp <= 9) {
    // query tile, while the load warps already stream K and V: row i holds
    // query m = qt * 64 + (i % nrow) of the kv group (head-major,
    // m = hl * wb + r), zero past m_total.  All of a thread's loads are
    // issued before its stores.
    constexpr int kFill = 288;                            // threads of warps 1..9
    constexpr int kPer = (128 * (D / 8) + kFill - 1) / kFill;
    const int t = tid - 32;
    uint4 v[kPer];
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int it = t + k * kFill;
      const int i = it / (D / 8), c = it - i * (D / 8);
      const int m = qt * TR + (i % nrow);
      v[k] = make_uint4(0u, 0u, 0u, 0u);
      if (it < 128 * (D / 8) && m < m_total) {
        const int hl = m / wb, r = m - hl * wb;
        v[k] = *reinterpret_cast<const uint4*>(
            p.q + (static_cast<size_t>(r0 + r) * p.Hq + g * p.group + hl) * D + c * 8);
      }
    }
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int it = t + k * kFill;
      const int i = it / (D / 8), c = it - i * (D / 8);
      if (it < 128 * (D / 8))
        *reinterpret_cast<uint4*>(smem + L::kQ + (c >> 3) * 16384 + swz(i, c & 7)) = v[k];
    }
    fence_async_smem();  // the MMAs read the tile through the async proxy
    __syncwarp();
    if (lane == 0) mbar_arrive(q_ready);
  }

  if (warp == 0 || warp == 10) {
    // ------------------------------------------------------------ TMA producers
    // Warp 0 loads the K steps, warp 10 the V steps, each into its own ring
    // as soon as a slot is free.  A step's second chunk past the split's end
    // is a load from beyond the cache, which TMA fills with zeros (finite V
    // for the masked keys).
    if (lane == 0 && nst > 0) {
      const bool is_k = warp == 0;
      const CUtensorMap* mc = is_k ? &tm_kc : &tm_vc;
      const CUtensorMap* mw = is_k ? &tm_kw : &tm_vw;
      uint64_t* fullb = is_k ? kfull : vfull;
      uint64_t* emptyb = is_k ? kempty : vempty;
      uint8_t* ring = smem + (is_k ? L::kK0 : L::kV0);
      const int y_oob = p.max_prefix > 0 ? p.max_prefix : 1;
      int n = 0;
      for (; n < nst; ++n) {
        const int s = n % kTcRing;
        if (n >= kTcRing &&
            !mbar_wait(&emptyb[s], static_cast<uint32_t>(n / kTcRing - 1) & 1u, p.limit_ns, abort))
          break;
        uint64_t* bar = &fullb[s];
        mbar_arrive_expect_tx(bar, 2u * NB * L::kBox);
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int k = 2 * n + half;
          const int c = c0 + k;
#pragma unroll
          for (int hf = 0; hf < NB; ++hf) {
            uint8_t* d = ring + s * L::kStep + hf * 16384 + half * L::kBox;
            if (k >= nmy)
              tma_load_4d(d, mc, bar, hf * 64, g, y_oob, b);
            else if (c < ncc)
              tma_load_4d(d, mc, bar, hf * 64, g, c * kAttnChunk, b);
            else if (c == ncc)
              tma_load_3d(d, mw, bar, hf * 64, g, r0);
            else
              tma_load_4d(d, mc, bar, hf * 64, g, S0 + (c - ncc - 1) * kAttnChunk, b);
          }
        }
      }
      if (n < nst) {
        if (!*abort) {
          *abort = 1;
          atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
        }
        // the copies in flight land before the CTA can exit
        for (int j = max(0, n - kTcRing); j < n; ++j)
          mbar_wait(&fullb[j % kTcRing], static_cast<uint32_t>(j / kTcRing) & 1u, p.limit_ns, nullptr);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA thread
    if (lane == 0 && nst > 0) {
      const uint32_t idesc_s = umma_idesc_bf16(128, 128);
      const uint32_t idesc_o = umma_idesc_bf16(128, D) | (1u << 16);  // B (V) MN-major
      // descriptors as 32-bit low words (start address >> 4, leading byte
      // offset) plus the high word they share (stride byte offset 1024,
      // version, 128-byte swizzle), advanced by immediates
      const uint32_t desc_hi = static_cast<uint32_t>(umma_desc_sw128(0) >> 32);
      const uint32_t q_lo = static_cast<uint32_t>(umma_desc_sw128(smem_u32(smem + L::kQ)));
      const uint32_t k0_lo = static_cast<uint32_t>(umma_desc_sw128(smem_u32(smem + L::kK0)));
      const uint32_t v0_lo = static_cast<uint32_t>(umma_desc_mn_sw128(smem_u32(smem + L::kV0), 16384));
      const uint32_t p_lo = static_cast<uint32_t>(umma_desc_sw128(smem_u32(smem + L::kP0)));
      // S(j) = Q K(j)^T into buffer j % 2, once K(j) has landed and the
      // softmax has read S(j - 2) out of that buffer
      auto qk = [&](int j) -> bool {
        const int s = j % kTcRing;
        if (!mbar_wait(&kfull[s], static_cast<uint32_t>(j / kTcRing) & 1u, p.limit_ns, abort))
          return false;
        if (j >= 2 && !mbar_wait(&s_free[j & 1], static_cast<uint32_t>((j - 2) >> 1) & 1u,
                                 p.limit_ns, abort))
          return false;
        tc_fence_after();
        const uint32_t k_lo = k0_lo + static_cast<uint32_t>(s) * (L::kStep >> 4);
        const uint32_t d = tmem + static_cast<uint32_t>((j & 1) * 128);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk)
          umma_bf16_lo(d, q_lo + static_cast<uint32_t>((kk >> 2) * (16384 >> 4) + (kk & 3) * 2),
                       k_lo + static_cast<uint32_t>((kk >> 2) * (16384 >> 4) + (kk & 3) * 2),
                       desc_hi, idesc_s, kk > 0 ? 1u : 0u);
        umma_commit(&s_full[j & 1]);
        umma_commit(&kempty[s]);
        return true;
      };
      bool ok = mbar_wait(q_ready, 0, p.limit_ns, abort);
      for (int j = 0; j < 2 && j < nst && ok; ++j) ok = qk(j);
      for (int i = 0; i < nst && ok; ++i) {
        const int s = i % kTcRing;
        if (!mbar_wait(p_full, static_cast<uint32_t>(i) & 1u, p.limit_ns, abort) ||
            !mbar_wait(&vfull[s], static_cast<uint32_t>(i / kTcRing) & 1u, p.limit_ns, abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t v_lo = v0_lo + static_cast<uint32_t>(s) * (L::kStep >> 4);
        const uint32_t d = tmem + 256u;
        const uint32_t acc0 = i != 0 ? 1u : 0u;
#pragma unroll
        for (int kk = 0; kk < kTcKeys / 16; ++kk)  // 16 keys per k-step
          umma_bf16_lo(d, p_lo + static_cast<uint32_t>((kk >> 2) * (16384 >> 4) + (kk & 3) * 2),
                       v_lo + static_cast<uint32_t>(kk * (2048 >> 4)), desc_hi, idesc_o,
                       kk != 0 ? 1u : acc0);
        umma_commit(pv_done);
        umma_commit(&vempty[s]);
        if (i + 2 < nst) ok = qk(i + 2);
      }
      if (!ok) {
        if (!*abort) {
          *abort = 1;
          atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
        }
        umma_commit(drain);  // completes once every MMA issued so far is done
        mbar_wait(drain, 0, p.limit_ns, nullptr);
      }
    }
  } else {
    // ------------------------------------------------------------ softmax
    // Warp w reads lane quadrant q = w % 4: query row qi = 32 rb + lane with
    // rb = q % (nrow / 32), and takes key group kg (of ngrp) of every step.
    // The warps of quadrants rb (high parts) and 2 + rb (low parts) own O.
    const int q = warp & 3, h = (warp - 2) >> 2;
    const int nrb = nrow / 32;
    const int rb = q % nrb;
    const int ngrp = 8 / nrb;
    const int kg = 2 * (q / nrb) + h;
    const int qi = rb * 32 + lane;
    const bool owner = q == rb || q == 2 + rb;
    const bool hi_owner = q == rb;
    const uint32_t lanes = tmem + (static_cast<uint32_t>(q * 32) << 16);
    const uint32_t bar_id = 1u + static_cast<uint32_t>(rb);
    const uint32_t bar_n = 32u * static_cast<uint32_t>(ngrp);
    const float sl2 = 1.4426950408889634f / sqrtf(static_cast<float>(D));  // log2(e)/sqrt(D)
    auto run = [&](auto kpg_c) {
      constexpr int KPG = decltype(kpg_c)::value;  // keys per warp and step
      float m_run = -INFINITY, l_run = 0.f;
      bool ok = true;
      const int k0 = kg * KPG;            // first key of this warp in a step
      const int half = k0 >> 6;           // its chunk within the step
      for (int i = 0; i < nst; ++i) {
        const int bb = i & 1;
        ok = ok && mbar_wait(&s_full[bb], static_cast<uint32_t>(i >> 1) & 1u, p.limit_ns, abort);
        ok = __all_sync(0xffffffffu, ok);
        float sv[KPG];
        float mx = -INFINITY;
        if (ok) {
          tc_fence_after();
          tmem_ld_cols<KPG>(lanes + static_cast<uint32_t>(bb * 128 + k0), sv);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&s_free[bb]);
          const int nv = nvalid(2 * i + half);
          if (nv >= kAttnChunk) {
#pragma unroll
            for (int j = 0; j < KPG; ++j) {
              sv[j] *= sl2;
              mx = fmaxf(mx, sv[j]);
            }
          } else {
#pragma unroll
            for (int j = 0; j < KPG; ++j) {
              sv[j] = ((k0 + j) & 63) < nv ? sv[j] * sl2 : -INFINITY;
              mx = fmaxf(mx, sv[j]);
            }
          }
        }
        xm[(bb * 8 + kg) * 64 + qi] = mx;
        ok = named_barrier_and(bar_id, bar_n, ok);  // the row's warps stop together
        if (!ok) break;
        float mc = -INFINITY;
        for (int q2 = 0; q2 < ngrp; ++q2) mc = fmaxf(mc, xm[(bb * 8 + q2) * 64 + qi]);
        float alpha = 1.f;
        const bool raise = mc > m_run + 8.f;
        if (raise) {
          alpha = ex2_approx(m_run - mc);  // 0 while m is still -inf
          m_run = mc;
          l_run *= alpha;
        }
        // P V of the previous step complete: O may be rescaled, P rewritten
        if (i > 0)
          ok = __all_sync(0xffffffffu, mbar_wait(pv_done, static_cast<uint32_t>(i - 1) & 1u,
                                                 p.limit_ns, abort));
        if (ok && owner && i > 0 && __any_sync(0xffffffffu, raise)) {
          tc_fence_after();
#pragma unroll
          for (int cc = 0; cc < HALF; cc += 32) {
            float o[32];
            const uint32_t ta = lanes + 256u + static_cast<uint32_t>(h * HALF + cc);
            tmem_ld_32x32b_x32(ta, o);
#pragma unroll
            for (int j = 0; j < 32; ++j) o[j] *= alpha;
            tmem_st_32x32b_x32(ta, o);
          }
          tc_fence_before();
        }
        float ls = 0.f;
#pragma unroll
        for (int j = 0; j < KPG; ++j) {
          sv[j] = ex2_approx(sv[j] - m_run);  // masked keys: exp2(-inf) = 0
          ls += sv[j];
        }
        l_run += ls;
        if (ok) {
          // keys k0..k0+KPG-1 of query qi: high parts in P row qi, low
          // parts in row 64 + qi; key block k0 / 64, 16-byte chunks from
          // (k0 % 64) / 8
          uint8_t* pb = smem + L::kP0 + half * 16384;
#pragma unroll
          for (int c = 0; c < KPG / 8; ++c) {
            uint32_t hw[4], lw[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) split_bf16x2(sv[8 * c + 2 * e], sv[8 * c + 2 * e + 1], hw[e], lw[e]);
            const int ch = ((k0 & 63) >> 3) + c;
            *reinterpret_cast<uint4*>(pb + swz(qi, ch)) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
            *reinterpret_cast<uint4*>(pb + swz(64 + qi, ch)) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
          }
          fence_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(p_full);
        } else if (lane == 0 && !*abort) {
          *abort = 1;
          atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
        }
      }
      // every P V is complete before O is read; the row sum is all groups'
      if (ok && nst > 0)
        ok = __all_sync(0xffffffffu, mbar_wait(pv_done, static_cast<uint32_t>(nst - 1) & 1u,
                                               p.limit_ns, abort));
      xl[kg * 64 + qi] = l_run;
      ok = named_barrier_and(bar_id, bar_n, ok);
      float l_tot = 0.f;
      for (int q2 = 0; q2 < ngrp; ++q2) l_tot += xl[q2 * 64 + qi];
      tc_fence_after();
      // Both halves of O to shared memory -- the K and V rings, free now
      // that every MMA has completed -- as [2][64][D + 4] (rows padded so
      // that the lanes' 16-byte stores fall in distinct banks), then whole
      // rows to global memory, one 512-byte row per warp instruction.
      constexpr int LDC = D + 4;
      float* comb = reinterpret_cast<float*>(smem + L::kK0);
      float* rowinfo = comb + 2 * 64 * LDC;  // [64] (m, l)
      if (ok && owner) {  // warp-uniform: the TMEM loads are warp-collective
        float* dc = comb + ((hi_owner ? 0 : 64) + qi) * LDC + h * HALF;
#pragma unroll
        for (int cc = 0; cc < HALF; cc += 32) {
          float o[32];
          if (nst > 0)
            tmem_ld_32x32b_x32(lanes + 256u + static_cast<uint32_t>(h * HALF + cc), o);
          else
#pragma unroll
            for (int j = 0; j < 32; ++j) o[j] = 0.f;  // a split without keys
#pragma unroll
          for (int j = 0; j < 32; j += 4)
            *reinterpret_cast<float4*>(dc + cc + j) = make_float4(o[j], o[j + 1], o[j + 2], o[j + 3]);
        }
        if (hi_owner && h == 0) *reinterpret_cast<float2*>(rowinfo + 2 * qi) = make_float2(m_run, l_tot);
      }
      ok = named_barrier_and(5, 256, ok);  // every softmax warp
      if (ok) {
        const int rows_here = min(TR, m_tile);
        for (int r = warp - 2; r < rows_here; r += 8) {
          if (lane >= D / 4) continue;
          const float4 hv = *reinterpret_cast<const float4*>(comb + r * LDC + 4 * lane);
          const float4 lv = *reinterpret_cast<const float4*>(comb + (64 + r) * LDC + 4 * lane);
          const float2 ml = *reinterpret_cast<const float2*>(rowinfo + 2 * r);
          float4 o4 = make_float4(hv.x + lv.x, hv.y + lv.y, hv.z + lv.z, hv.w + lv.w);
          if (p.splits == 1) {
            const float sc = ml.y > 0.f ? 1.0f / ml.y : 0.f;
            o4 = make_float4(o4.x * sc, o4.y * sc, o4.z * sc, o4.w * sc);
            const int m = qt * TR + r;
            const int hl = m / wb, rr = m - hl * wb;
            if (in_bounds(r0 + rr, p.R, p.status))
              *reinterpret_cast<float4*>(p.out + (static_cast<size_t>(r0 + rr) * p.Hq + g * p.group + hl) * D +
                                         4 * lane) = o4;
          } else {
            const size_t pr = (static_cast<size_t>(slot) * p.splits + split) * TR + r;
            *reinterpret_cast<float4*>(p.part + pr * D + 4 * lane) = o4;
            if (lane == 0) *reinterpret_cast<float2*>(p.part_ml + pr * 2) = ml;
          }
        }
      } else if (lane == 0 && !*abort) {
        *abort = 1;
        atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
      }
    };
    if (nrow == 32)
      run(std::integral_constant<int, 16>{});
    else
      run(std::integral_constant<int, 32>{});
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTcTmemCols);
  }
  if (p.splits == 1 || *abort) return;

  // the last CTA of the slot combines the splits' partials, as in the
  // mma.sync kernel
  __threadfence();
  __syncthreads();
  if (tid == 0) *s_flag = (atomicAdd(&p.tickets[slot], 1) == p.splits - 1);
  __syncthreads();
  if (!*s_flag) return;
  __threadfence();
  __shared__ float s_w[TR][kMaxAttnSplits];
  const float* bo = p.part + static_cast<size_t>(slot) * p.splits * TR * D;
  const float* bml = p.part_ml + static_cast<size_t>(slot) * p.splits * TR * 2;
  const int rows_here = min(TR, m_tile);
  for (int r = tid; r < rows_here; r += blockDim.x) {
    float M = -INFINITY;
    for (int sp = 0; sp < p.splits; ++sp) M = fmaxf(M, __ldcg(bml + (sp * TR + r) * 2));
    float Lsum = 0.f;
    for (int sp = 0; sp < p.splits; ++sp) {
      const float2 v = __ldcg(reinterpret_cast<const float2*>(bml + (sp * TR + r) * 2));
      const float wgt = v.x == -INFINITY ? 0.f : exp2f(v.x - M);
      s_w[r][sp] = wgt;
      Lsum += wgt * v.y;
    }
    const float inv = Lsum > 0.f ? 1.0f / Lsum : 0.f;
    for (int sp = 0; sp < p.splits; ++sp) s_w[r][sp] *= inv;
  }
  __syncthreads();
  constexpr int D4 = D / 4;
  for (int it = tid; it < rows_here * D4; it += blockDim.x) {
    const int r = it / D4, d = (it - r * D4) * 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int sp = 0; sp < kMaxAttnSplits; ++sp) {
      if (sp < p.splits) {
        const float4 v = __ldcg(reinterpret_cast<const float4*>(
            bo + (static_cast<size_t>(sp) * TR + r) * D + d));
        const float wgt = s_w[r][sp];
        acc.x = fmaf(wgt, v.x, acc.x);
        acc.y = fmaf(wgt, v.y, acc.y);
        acc.z = fmaf(wgt, v.z, acc.z);
        acc.w = fmaf(wgt, v.w, acc.w);
      }
    }
    const int m = qt * TR + r;
    const int hl = m / wb, rr = m - hl * wb;
    if (in_bounds(r0 + rr, p.R, p.status))
      *reinterpret_cast<float4*>(p.out + (static_cast<size_t>(r0 + rr) * p.Hq + g * p.group + hl) * D + d) = acc;
  }
  if (tid == 0) p.tickets[slot] = 0;
}

// ------------------------------------------------------------------ cache append
// Prefix-cache append on commit (Sec. 6.3): window row r (blockIdx.x) of its
// sequence, if committed after the step (mask 0), is copied 16 bytes per
// thread into the cache at its absolute position; positions outside the
// cache are skipped.
__global__ void __launch_bounds__(256)
    kv_append_kernel(uint4* __restrict__ k_cache, uint4* __restrict__ v_cache,
                     const uint4* __restrict__ k_win, const uint4* __restrict__ v_win,
                     const int* __restrict__ cu_rows, const int* __restrict__ row_pos,
                     const uint8_t* __restrict__ mask, int B, int Pmax, int vec_per_row) {
  // launched as a programmatic dependent of the attention, which completes
  // only after the decision: the mask read below is final
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int r = blockIdx.x;
  if (mask[r] != 0) return;
  const int pos = row_pos[r];
  if (pos < 0 || pos >= Pmax) return;
  int b = 0;
  while (b + 1 < B && cu_rows[b + 1] <= r) ++b;
  const size_t dst = (static_cast<size_t>(b) * Pmax + pos) * vec_per_row;
  const size_t src = static_cast<size_t>(r) * vec_per_row;
  for (int i = threadIdx.x; i < vec_per_row; i += blockDim.x) {
    k_cache[dst + i] = k_win[src + i];
    v_cache[dst + i] = v_win[src + i];
  }
}

cudaError_t launch_kv_append(uint16_t* k_cache, uint16_t* v_cache, const uint16_t* k_win,
                             const uint16_t* v_win, const int* cu_rows, const int* row_pos,
                             const uint8_t* mask, int B, int rows, int Pmax, int hkvd,
                             cudaStream_t st, bool pdl) {
  if (rows <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(rows, 1, 1);
  cfg.blockDim = dim3(256, 1, 1);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kv_append_kernel, reinterpret_cast<uint4*>(k_cache),
                            reinterpret_cast<uint4*>(v_cache), reinterpret_cast<const uint4*>(k_win),
                            reinterpret_cast<const uint4*>(v_win), cu_rows, row_pos, mask, B, Pmax,
                            hkvd / 8);
}

// q and the window K/V copied in by another stream (a copy engine), which
// then writes the step's ticket to *p.ready: thread 0 polls it with an
// acquire at system scope, with a time limit; on timeout the CTA records
// EBD_ERR_TIMEOUT and does no work.
__device__ __forceinline__ bool wait_ready(const AttnParams& p) {
  __shared__ int s_ok;
  if (threadIdx.x == 0) {
    auto seen = [&]() {
      unsigned v;
      asm volatile("ld.acquire.sys.global.u32 %0, [%1];" : "=r"(v) : "l"(p.ready) : "memory");
      return v == p.ready_ticket;
    };
    bool ok = seen();
    if (!ok) {
      const uint64_t t0 = global_timer_ns();
      while (!(ok = seen()) && global_timer_ns() - t0 <= p.limit_ns) __nanosleep(200);
    }
    if (ok)
      asm volatile("fence.proxy.async.global;" ::: "memory");  // the TMA reads of the window K/V
    else
      atomicCAS(p.status, 0, EBD_ERR_TIMEOUT);
    s_ok = ok ? 1 : 0;
  }
  __syncthreads();
  return s_ok != 0;
}

// The whole kernel; with p.wait_prior every CTA, whichever way it finishes,
// waits for the grid it is a programmatic dependent of (the decision) before
// it exits, so that a kernel launched after this one as its dependent sees
// that grid complete as well.
template <int D>
__global__ void __launch_bounds__(kAttnThreads)
    attn_kernel(const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
                const __grid_constant__ CUtensorMap tm_kw, const __grid_constant__ CUtensorMap tm_vw,
                const AttnParams p) {
  if (p.ready == nullptr || wait_ready(p)) attn_body<D>(tm_kc, tm_vc, tm_kw, tm_vw, p);
  if (p.wait_prior) asm volatile("griddepcontrol.wait;" ::: "memory");
}

template <int D>
__global__ void __launch_bounds__(kAttnTcThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
                   const __grid_constant__ CUtensorMap tm_kw, const __grid_constant__ CUtensorMap tm_vw,
                   const AttnParams p) {
  if (p.ready == nullptr || wait_ready(p)) attn_tc_body<D>(tm_kc, tm_vc, tm_kw, tm_vw, p);
  if (p.wait_prior) asm volatile("griddepcontrol.wait;" ::: "memory");
}

cudaError_t attn_configure() {
  const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
  const int bytes = kAttnStages * kStageBytes + 1024 + 64;
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(attn_kernel<64>, a, bytes)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(attn_kernel<128>, a, bytes)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(attn_tc_kernel<64>, a, TcMap<64>::kDyn)) != cudaSuccess) return e;
  return cudaFuncSetAttribute(attn_tc_kernel<128>, a, TcMap<128>::kDyn);
}

cudaError_t launch_attention(const CUtensorMap& kc, const CUtensorMap& vc, const CUtensorMap& kw,
                             const CUtensorMap& vw, const AttnParams& p, cudaStream_t st,
                             bool pdl) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(p.splits, p.max_qtiles, p.B * p.Hkv);
  cfg.blockDim = dim3(p.tc ? kAttnTcThreads : kAttnThreads, 1, 1);
  cfg.dynamicSmemBytes = p.tc ? (p.D == 64 ? TcMap<64>::kDyn : TcMap<128>::kDyn)
                              : kAttnStages * kStageBytes + 1024 + 64;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (p.tc)
    return p.D == 64 ? cudaLaunchKernelEx(&cfg, attn_tc_kernel<64>, kc, vc, kw, vw, p)
                     : cudaLaunchKernelEx(&cfg, attn_tc_kernel<128>, kc, vc, kw, vw, p);
  if (p.D == 64) return cudaLaunchKernelEx(&cfg, attn_kernel<64>, kc, vc, kw, vw, p);
  return cudaLaunchKernelEx(&cfg, attn_kernel<128>, kc, vc, kw, vw, p);
}

}  // namespace ebd
