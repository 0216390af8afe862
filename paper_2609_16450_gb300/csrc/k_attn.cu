// Window attention: the active window's queries attend, without a mask, to
// the sequence's cached prefix keys, the window's own keys and, with a dual
// cache, a cached suffix range (bidirectional dLLM, Sec. 3; prefix and dual
// cache at the block boundaries, Sec. 6.3).
//   O = softmax(Q K^T / sqrt(D)) V, fp32 output.
// The key range is a list of 64-key chunks: prefix tiles of the cache, one
// tile of window rows, then suffix tiles of the cache.
//
// Grid: (key split, query tile, sequence x kv head).  A query tile is 64 rows
// of (query head of the kv group, window row); each of the 4 warps owns 16
// rows.  K/V tiles of 64 keys are staged by TMA (128-byte swizzle) through a
// 3-stage ring; Q K^T runs on mma.sync bf16 with fp32 accumulation; the
// probabilities are split into a bf16 high part and a bf16 remainder so that
// P V keeps ~16 mantissa bits.  Splits of the key range combine their
// (max, sum, O) partials in the last CTA to finish (atomic ticket).
#include "internal.h"
#include "ptx.cuh"

namespace ebd {

namespace {

constexpr int kStageBytes = 4 * 8192;  // K and V, two 64-dim halves each

// byte offset of 16-byte chunk `c` (0..7) of row `r` in a 128B-swizzled tile
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return static_cast<uint32_t>(r * 128 + ((c ^ (r & 7)) << 4));
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

cudaError_t attn_configure() {
  const int bytes = kAttnStages * kStageBytes + 1024 + 64;
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

cudaError_t launch_attention(const CUtensorMap& kc, const CUtensorMap& vc, const CUtensorMap& kw,
                             const CUtensorMap& vw, const AttnParams& p, cudaStream_t st,
                             bool pdl) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(p.splits, p.max_qtiles, p.B * p.Hkv);
  cfg.blockDim = dim3(kAttnThreads, 1, 1);
  cfg.dynamicSmemBytes = kAttnStages * kStageBytes + 1024 + 64;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (p.D == 64) return cudaLaunchKernelEx(&cfg, attn_kernel<64>, kc, vc, kw, vw, p);
  return cudaLaunchKernelEx(&cfg, attn_kernel<128>, kc, vc, kw, vw, p);
}

}  // namespace ebd
