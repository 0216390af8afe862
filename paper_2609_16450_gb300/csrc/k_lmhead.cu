// LM head fused with the softmax statistics of every window row.
//
// For each window row r and vocabulary entry v the logit is
// l[r][v] = sum_k h[r][k] W[v][k]; the kernel never stores it.  Each CTA owns a
// contiguous range of 64-row vocabulary units and keeps, per window row, the
// online-softmax state over the vocabulary it has seen:
//   m  = max logit,  S = sum exp(l - m),  T = sum exp(l - m) (l - m),
//   l2 = second largest logit (duplicates count),  idx = argmax (lowest).
// The decision kernel merges the per-CTA states into kappa = 1/S,
// H = ln S - T/S, Delta = (1 - exp(l2 - m)) / S and x_hat = idx, i.e. the
// statistics of App. B (Eq. app-confidence), Sec. 5.1 and Sec. 5.2.
//
// Tensor-core mapping (swap-AB): the vocabulary tile is the MMA's M = 128
// (A = W rows, K-major, streamed by TMA with an evict-first L2 policy), the
// window rows are N (B = hidden rows, K-major), the fp32 accumulator lives
// in TMEM as 128 lanes (vocabulary) x N columns (rows).  Warp 0 issues TMA,
// warp 1 issues tcgen05.mma, warps 2..5 (and 6..9) drain TMEM and run the
// statistics.  Where the rows make the tensor cores the bound, CTA pairs run
// cta_group::2 MMAs with M = 256 (two SMs, one accumulator tile).
#include <climits>
#include <cstdlib>

#include "internal.h"
#include "ptx.cuh"

namespace ebd {

namespace {

constexpr uint32_t kATile = 128 * 128;  // 128 rows x 64 bf16
constexpr int kTLd = 132;               // transpose buffer row stride (floats)
constexpr uint32_t kTBytes = 32 * kTLd * 4;  // transpose buffer of one epilogue warpgroup

__device__ __forceinline__ void state_merge(float& m, float& s, float& t, float& l2, int& idx,
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
  if (bm == -INFINITY) return;  // the other side is empty
  const float dl = bm - m;      // <= 0
  const float sc = __expf(dl);
  t = t + sc * (bt + dl * bs);
  s = s + sc * bs;
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

// MMAs of one pipeline stage: KBS k-boxes x 4 k16 steps x NSUB N sub-tiles,
// descriptors advanced by immediates (k16 step = 32 bytes = 2 in the
// descriptor's address field; k-box = kATile bytes of A, b_step of B; N
// sub-tile sb at sb * sub_desc of B and sb * sub_cols TMEM columns).
template <int KBS, int NSUB, bool PAIR>
__device__ __forceinline__ void mma_stage(uint32_t d, uint32_t a_lo, uint32_t b_lo,
                                          uint32_t b_step, uint32_t sub_desc, uint32_t sub_cols,
                                          uint32_t hi, uint32_t idesc, uint32_t acc0) {
#pragma unroll
  for (int j = 0; j < KBS; ++j)
#pragma unroll
    for (int kk = 0; kk < 4; ++kk)
#pragma unroll
      for (int sb = 0; sb < NSUB; ++sb) {
        const uint32_t dd = d + static_cast<uint32_t>(sb) * sub_cols;
        const uint32_t al = a_lo + static_cast<uint32_t>(j * (kATile >> 4) + kk * 2);
        const uint32_t bl = b_lo + static_cast<uint32_t>(j) * b_step +
                            static_cast<uint32_t>(sb) * sub_desc + static_cast<uint32_t>(kk * 2);
        if (PAIR)
          umma_bf16_lo_pair(dd, al, bl, hi, idesc, (j | kk) != 0 ? 1u : acc0);
        else
          umma_bf16_lo(dd, al, bl, hi, idesc, (j | kk) != 0 ? 1u : acc0);
      }
}

// Waits with a back-off between polls: for warps whose wait is long and not
// latency-critical, so that they leave the issue slots of their SM
// sub-partition to the producer and MMA threads.
__device__ __forceinline__ bool mbar_wait_sleepy(uint64_t* bar, uint32_t parity, uint64_t limit_ns,
                                                 volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (;;) {
    __nanosleep(256);
    if (mbar_try_wait(bar, parity)) return true;
    if (abort != nullptr && *abort) return false;
    if (global_timer_ns() - t0 > limit_ns) return false;
  }
}

__device__ __forceinline__ void record_error(int* status, volatile int* abort, int code) {
  *abort = 1;
  atomicCAS(status, 0, code);
}

// Statistics of one accumulator buffer by one epilogue warpgroup, in slices
// of 32 columns (window rows): each slice goes TMEM -> registers -> a
// transpose in shared memory, after which 4 threads share a column and scan
// its 128 vocabulary lanes (32 each); the column's state is merged into the
// running state of its row.  `release` is called once this thread has
// loaded its last slice (the MMAs may then overwrite the buffer).  Returns
// whether it was called.
template <typename Release>
__device__ __forceinline__ bool epilogue_buffer(uint32_t taddr0, int wg, int nwg, int n_pad,
                                                float* sTw, int lanev, int et, uint32_t bar_id,
                                                int vbase, int valid, float* st_m, float* st_s,
                                                float* st_t, float* st_l2, int* st_i,
                                                Release release) {
  bool released = false;
  const bool lv = lanev < valid;
  for (int cc = 32 * wg; cc < n_pad; cc += 32 * nwg) {
    float v[32];
    if (n_pad - cc >= 32)
      tmem_ld_32x32b_x32(taddr0 + static_cast<uint32_t>(cc), v);
    else
      tmem_ld_32x32b_x16(taddr0 + static_cast<uint32_t>(cc), v);
    if (cc + 32 * nwg >= n_pad) {  // this warpgroup's last slice is in registers
      release();
      released = true;
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) sTw[j * kTLd + lanev] = lv ? v[j] : -INFINITY;
    named_barrier(bar_id, 128);
    {
      const int j = et >> 2, q = et & 3;
      float x[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) x[i] = sTw[j * kTLd + q + 4 * i];
      // branch-free scan: the threads of a warp see different data
      float m = -INFINITY, l2 = -INFINITY;
      int ii = -1;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        l2 = fmaxf(l2, fminf(m, x[i]));
        ii = x[i] > m ? i : ii;  // strict: the first (lowest) index of the maximum
        m = fmaxf(m, x[i]);
      }
      int idx = ii < 0 ? INT_MAX : vbase + q + 4 * ii;  // vbase includes the shard offset
      float s = 0.f, t = 0.f;
      if (m != -INFINITY) {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float dl = x[i] - m;
          const float e = __expf(dl);
          s += e;
          t = fmaf(e, e > 0.f ? dl : 0.f, t);  // masked lanes: e = 0, dl = -inf
        }
      }
#pragma unroll
      for (int off = 1; off <= 2; off <<= 1) {
        const float bm = __shfl_xor_sync(0xffffffffu, m, off);
        const float bs = __shfl_xor_sync(0xffffffffu, s, off);
        const float bt = __shfl_xor_sync(0xffffffffu, t, off);
        const float bl = __shfl_xor_sync(0xffffffffu, l2, off);
        const int bi = __shfl_xor_sync(0xffffffffu, idx, off);
        state_merge(m, s, t, l2, idx, bm, bs, bt, bl, bi);
      }
      const int r = cc + j;
      if (q == 0 && r < n_pad) {
        float M = st_m[r], S = st_s[r], T = st_t[r], L2 = st_l2[r];
        int I = st_i[r];
        state_merge(M, S, T, L2, I, m, s, t, l2, idx);
        st_m[r] = M;
        st_s[r] = S;
        st_t[r] = T;
        st_l2[r] = L2;
        st_i[r] = I;
      }
    }
    named_barrier(bar_id, 128);
  }
  return released;
}

}  // namespace

// PAIR (p.pair) and PACKED (p.packed) are template parameters: a runtime
// branch in the single-thread producer or MMA loop costs measurable time.
//
// PAIR: the CTAs of a cluster of 2 form a pair that runs cta_group::2 MMAs
// of M = 256 vocabulary rows.  A vocabulary chunk is 4 units: the even CTA
// (the leader) loads units 0-1 of it, the odd CTA units 2-3, each into its
// own shared memory; each loads its half of every N sub-tile of hidden rows.
// The leader's thread issues the MMAs, whose 256 x N accumulator lands as
// 128 lanes x N columns in each CTA's TMEM, and its commits arrive on both
// CTAs' barriers.  Both CTAs' copies complete on the leader's stage
// barriers; both epilogues release the accumulator on the leader's barrier.
// Each SM thus receives half of the hidden rows per MMA, which halves the
// operand bytes per flop against a 128-row tile over the same rows.
//
// Row groups (p.rgroups = 2, paired launches of more than 432 rows): pair q
// serves rows [row0 + g nb, row0 + (g + 1) nb) of group g = q / nwork over
// the vocabulary range of owner q % nwork, and writes its partials to
// columns [0, grp_cols) of those rows.
template <bool PAIR, bool PACKED>
__global__ void __launch_bounds__(kLmThreads, 1)
    lm_stats_kernel(const __grid_constant__ CUtensorMap tmap_w,
                    const __grid_constant__ CUtensorMap tmap_h, const LmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem + p.off_a;
  uint8_t* sB = smem + p.off_b;
  float* sT = reinterpret_cast<float*>(smem + p.off_t);
  float* st_m = reinterpret_cast<float*>(smem + p.off_st);
  float* st_s = st_m + p.n_pad;
  float* st_t = st_s + p.n_pad;
  float* st_l2 = st_t + p.n_pad;
  int* st_i = reinterpret_cast<int*>(st_l2 + p.n_pad);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + p.off_bar);
  uint64_t* full = bars;
  uint64_t* empty = bars + p.stages;
  uint64_t* acc_full = bars + 2 * p.stages;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* drain = acc_empty + 2;
  uint64_t* dummy = drain + 1;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(dummy + 1);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_holder + 1);

  constexpr int kChunkUnits = PAIR ? 4 : 2;  // vocabulary units per accumulator
  const int tid = threadIdx.x;
  const int warp = __shfl_sync(0xffffffffu, tid / 32, 0);
  const int lane = tid & 31;
  const uint32_t crank = PAIR ? cluster_ctarank() : 0u;
  const bool leader = crank == 0;
  // row group of this CTA (its pair) and its owner index within the group
  const int q = PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int grp = q / p.nwork;
  const int owner = q - grp * p.nwork;
  const int rbase = p.row0 + grp * p.nb;                 // first row of the group
  const int rows_g = min(p.rgroups > 1 ? p.nb : p.rows, p.rows - grp * p.nb);
  const int col = PAIR ? 2 * owner + static_cast<int>(crank) : owner;  // partial column
  // hidden rows of one N sub-tile that this CTA holds: all of them, or its
  // half in a pair
  const int hrows = PAIR ? p.nb / 2 : p.nb;

  if (tid == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], (PAIR ? 2 : 1) * 128 * p.nwg);  // both CTAs' epilogues
    }
    mbar_init(drain, 1);
    mbar_init(dummy, 1);
    *abort = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmap_w);
    tma_prefetch_desc(&tmap_h);
  }
  if (warp == 1) {
    if (PAIR)
      tmem_alloc_pair(tmem_holder, p.tmem_cols);
    else
      tmem_alloc(tmem_holder, p.tmem_cols);
  }
  if (tid >= 64) {
    for (int r = tid - 64; r < p.n_pad; r += kLmThreads - 64) {
      st_m[r] = -INFINITY;
      st_s[r] = 0.f;
      st_t[r] = 0.f;
      st_l2[r] = -INFINITY;
      st_i[r] = INT_MAX;
    }
  }
  tc_fence_before();
  if (PAIR)
    cluster_sync_all();  // the peer's barriers exist before anything arrives on them
  else
    __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;

  const int u0 = static_cast<int>((static_cast<long long>(owner) * p.n_units) / p.nwork);
  const int u1 = static_cast<int>((static_cast<long long>(owner + 1) * p.n_units) / p.nwork);
  const uint32_t b_sub = static_cast<uint32_t>(p.nsub * hrows) * 128u;  // one k-box of hidden rows here
  const uint32_t a_stage = static_cast<uint32_t>(p.kbs) * kATile;
  const uint32_t b_stage = static_cast<uint32_t>(p.kbs) * b_sub;
  // W units of a chunk that this CTA loads and accumulates: [ulo, ulo + 2)
  const int ulo = PAIR ? 2 * static_cast<int>(crank) : 0;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const uint64_t pol_w = l2_policy_evict_first();
      const uint64_t pol_h = l2_policy_evict_last();
      auto load = [&](void* dst, const CUtensorMap* map, int s, int x, int y, uint64_t pol) {
        if (PAIR)
          tma_load_2d_pair(dst, map, mapa_shared(smem_u32(&full[s]), 0), x, y, pol);
        else
          tma_load_2d(dst, map, &full[s], x, y, pol);
      };
      auto load4 = [&](void* dst, const CUtensorMap* map, int s, int z, int w, uint64_t pol) {
        tma_load_4d_pair(dst, map, mapa_shared(smem_u32(&full[s]), 0), 0, 0, z, w, pol);
      };
      // stage fill: vocabulary chunk u (kChunkUnits units), k-stage ks; the
      // leader arms the stage for the W and hidden bytes of both CTAs.
      // A pair reads packed W as a 4-D tensor (column, row, unit, k-box):
      // one box of two units by the stage's kbs k-boxes is a CTA's 128 W
      // rows of the whole stage in one copy, laid out as the MMAs read it
      // (the copies, not L2, set the paired kernel's operand feed: at 64 x 32
      // rows the LM head took 1522 us with two 8 KB boxes per k-box, 1394 us
      // with one 16 KB box, 1317 us with one box per stage).  A CTA with one
      // unit of the chunk still reads two (the second is the next pair's, or
      // zeros past the last unit) and its epilogue ignores the second.
      // Unpaired, HBM-bound launches read one unit at a time.
      auto issue_w = [&](int u, int ks, int s) {
        const int nu = min(kChunkUnits, u1 - u);
        const int nsubk = min(p.kbs, p.nkb - ks * p.kbs);
        // W bytes of the stage: one box of kbs k-boxes by two units per CTA
        // with units in the chunk (a stage past the last k-box reads zeros)
        const uint32_t w_bytes = (PACKED && PAIR)
                                     ? (nu > 2 ? 2u : 1u) * static_cast<uint32_t>(p.kbs) * kATile
                                     : static_cast<uint32_t>(nsubk * nu) * kUnit * 128u;
        if (leader)
          mbar_arrive_expect_tx(&full[s], w_bytes + static_cast<uint32_t>(nsubk * p.n_pad) * 128u);
        uint8_t* a_st = sA + static_cast<size_t>(s) * a_stage;
        if (PACKED && PAIR) {
          if (nu > ulo) load4(a_st, &tmap_w, s, u + ulo, ks * p.kbs, pol_w);
        } else {
          // one unit at a time, its k-boxes back to back: each W row is
          // requested as one contiguous run of nsubk * 128 bytes
          for (int ui = ulo; ui < min(ulo + 2, nu); ++ui) {
            for (int j = 0; j < nsubk; ++j) {
              const int x = PACKED ? 0 : (ks * p.kbs + j) * 64;
              const int y = PACKED ? ((u + ui) * p.nkb + ks * p.kbs + j) * kUnit : (u + ui) * kUnit;
              load(a_st + j * kATile + (ui - ulo) * (kUnit * 128), &tmap_w, s, x, y, pol_w);
            }
          }
        }
      };
      auto issue_h = [&](int ks, int s) {
        const int nsubk = min(p.kbs, p.nkb - ks * p.kbs);
        uint8_t* b_st = sB + static_cast<size_t>(s) * b_stage;
        for (int j = 0; j < nsubk; ++j)
          for (int sb = 0; sb < p.nsub; ++sb)
            load(b_st + j * b_sub + sb * hrows * 128, &tmap_h, s, (ks * p.kbs + j) * 64,
                 rbase + sb * p.nb + static_cast<int>(crank) * hrows, pol_h);
      };
      int u = u0, ks = 0;  // the next stage fill
      auto advance = [&]() {
        if (++ks == p.nks) {
          ks = 0;
          u += kChunkUnits;
        }
      };
      // The first stages' W go out before anything else.  As a programmatic
      // dependent of the copy of its hidden rows (ebd_step_host), the grid
      // waits for that copy only then; and only then does it release the
      // decision kernel, launched after it as a programmatic dependent,
      // which reads the decode state the same copy brings at once (and waits
      // for this grid's completion before it reads the partial states).
      // Released this late in every launch, the decision and the attention
      // after it no longer take SMs while this grid starts: LLaDA-8B step
      // 205.8 us (p90 213.5) with the release at kernel entry, 198.8 us
      // (p90 199.2) here; the LM head alone 155.7 against 156.0 us.
      int it = 0;
      {
        const int ks0 = ks;
        for (; it < p.stages && u < u1; ++it, advance()) issue_w(u, ks, it);  // stages start empty
        asm volatile("griddepcontrol.wait;" ::: "memory");
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        for (int i = 0, hk = ks0; i < it; ++i) {
          issue_h(hk, i);
          if (++hk == p.nks) hk = 0;
        }
      }
      int s = it == p.stages ? 0 : it;        // stage of iteration it
      uint32_t ph = it == p.stages ? 1u : 0u;  // its phase parity
      bool ok = true;
      for (; u < u1; ++it, advance()) {
        if (!mbar_wait(&empty[s], ph ^ 1u, p.limit_ns, abort)) {
          ok = false;
          break;
        }
        issue_w(u, ks, s);
        issue_h(ks, s);
        if (++s == p.stages) {
          s = 0;
          ph ^= 1u;
        }
      }
      if (!ok) {
        if (!*abort) record_error(p.status, abort, EBD_ERR_TIMEOUT);
        if (leader) {
          // let the copies already in flight land before the CTA can exit
          for (int j = max(0, it - p.stages); j < it; ++j)
            mbar_wait(&full[j % p.stages], static_cast<uint32_t>(j / p.stages) & 1u, p.limit_ns,
                      nullptr);
        } else {
          // the peer's copies complete on the leader's barriers: give those
          // in flight time to land (a stage lands in a few microseconds)
          const uint64_t t0 = global_timer_ns();
          while (global_timer_ns() - t0 < 200ull * 1000) __nanosleep(1000);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && leader) {
      const uint32_t idesc = umma_idesc_bf16(PAIR ? 256 : 128, static_cast<uint32_t>(p.nb));
      const uint32_t desc_hi = static_cast<uint32_t>(umma_desc_sw128(0) >> 32);
      int it = 0, c = 0;
      int s = 0;        // stage of iteration it, as in the producer
      uint32_t ph = 0;
      bool ok = true;
      auto commit_stage = [&](int st) {
        if (PAIR)
          umma_commit_pair_mc(&empty[st], 0x3);
        else
          umma_commit(&empty[st]);
      };
      for (int u = u0; u < u1 && ok; u += kChunkUnits, ++c) {
        const int buf = c % p.nbuf;
        const uint32_t bph = static_cast<uint32_t>(c / p.nbuf) & 1u;
        if (!mbar_wait(&acc_empty[buf], bph ^ 1u, p.limit_ns, abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d0 = tmem_base + static_cast<uint32_t>(buf * p.acc_stride);
        for (int ks = 0; ks < p.nks; ++ks) {
          if (!mbar_wait(&full[s], ph, p.limit_ns, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int nsubk = min(p.kbs, p.nkb - ks * p.kbs);
          const uint32_t a_addr = smem_u32(sA + static_cast<size_t>(s) * a_stage);
          const uint32_t b_addr = smem_u32(sB + static_cast<size_t>(s) * b_stage);
          if (p.nsub <= 2 && nsubk >= 1 && nsubk <= 5) {
            // the unrolled issue path
            const uint32_t a_lo = static_cast<uint32_t>(umma_desc_sw128(a_addr));
            const uint32_t b_lo = static_cast<uint32_t>(umma_desc_sw128(b_addr));
            const uint32_t b_step = b_sub >> 4;
            const uint32_t sub_desc = static_cast<uint32_t>(hrows) * 8u;  // hrows x 128 B >> 4
            const uint32_t sub_cols = static_cast<uint32_t>(p.nb);
            const uint32_t acc0 = ks != 0 ? 1u : 0u;
#define EBD_STAGE(K, S) \
  mma_stage<K, S, PAIR>(d0, a_lo, b_lo, b_step, sub_desc, sub_cols, desc_hi, idesc, acc0)
            if (p.nsub == 1) {
              switch (nsubk) {
                case 1: EBD_STAGE(1, 1); break;
                case 2: EBD_STAGE(2, 1); break;
                case 3: EBD_STAGE(3, 1); break;
                case 4: EBD_STAGE(4, 1); break;
                default: EBD_STAGE(5, 1); break;
              }
            } else {
              switch (nsubk) {
                case 1: EBD_STAGE(1, 2); break;
                case 2: EBD_STAGE(2, 2); break;
                case 3: EBD_STAGE(3, 2); break;
                case 4: EBD_STAGE(4, 2); break;
                default: EBD_STAGE(5, 2); break;
              }
            }
#undef EBD_STAGE
          } else {
            for (int j = 0; j < nsubk; ++j) {
#pragma unroll
              for (int kk = 0; kk < 4; ++kk) {
                const uint64_t ad = umma_desc_sw128(a_addr + j * kATile + kk * 32);
                for (int sb = 0; sb < p.nsub; ++sb) {
                  const uint64_t bd = umma_desc_sw128(b_addr + j * b_sub + sb * hrows * 128 + kk * 32);
                  const uint32_t acc = (ks | j | kk) != 0 ? 1u : 0u;
                  const uint32_t dd = d0 + static_cast<uint32_t>(sb * p.nb);
                  if (PAIR)
                    umma_bf16_lo_pair(dd, static_cast<uint32_t>(ad), static_cast<uint32_t>(bd),
                                      desc_hi, idesc, acc);
                  else
                    umma_bf16(dd, ad, bd, idesc, acc);
                }
              }
            }
          }
          commit_stage(s);
          ++it;
          if (++s == p.stages) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        if (PAIR)
          umma_commit_pair_mc(&acc_full[buf], 0x3);
        else
          umma_commit(&acc_full[buf]);
      }
      if (!ok) {
        if (!*abort) record_error(p.status, abort, EBD_ERR_TIMEOUT);
        // completes once every MMA issued so far is done
        if (PAIR)
          umma_commit_pair(drain);
        else
          umma_commit(drain);
        mbar_wait(drain, 0, p.limit_ns, nullptr);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    // p.nwg warpgroups of 4 warps (one per TMEM lane quadrant) take the
    // 32-row column slices of the accumulator in turn; a second warpgroup
    // is used when the accumulator has a single buffer.
    const int wg = (tid - 64) >> 7;
    const int et = (tid - 64) & 127;  // thread within the warpgroup
    const int quad = warp & 3;        // TMEM lane quadrant this warp may read
    const int lanev = quad * 32 + lane;
    const uint32_t bar_id = 1u + static_cast<uint32_t>(wg);
    float* const sTw = sT + wg * (kTBytes / 4);
    bool ok = wg < p.nwg;
    if (ok && p.force_timeout) {
      ok = mbar_wait(dummy, 0, 20ull * 1000 * 1000, nullptr);
      ok = named_barrier_and(bar_id, 128, ok);
      if (!ok && et == 0 && wg == 0) record_error(p.status, abort, EBD_ERR_TIMEOUT);
    }
    const bool active = ok;
    auto release = [&](int buf) {  // this thread's reads of the accumulator are done
      tc_fence_before();
      if (PAIR)
        mbar_arrive_cluster(mapa_shared(smem_u32(&acc_empty[buf]), 0));
      else
        mbar_arrive(&acc_empty[buf]);
    };
    int c = 0;
    for (int u = u0; u < u1 && ok; u += kChunkUnits, ++c) {
      const int nu = min(kChunkUnits, u1 - u);
      const int buf = c % p.nbuf;
      const uint32_t bph = static_cast<uint32_t>(c / p.nbuf) & 1u;
      bool w = mbar_wait_sleepy(&acc_full[buf], bph, p.limit_ns, abort);
      ok = named_barrier_and(bar_id, 128, w);
      if (!ok) {
        if (et == 0 && !*abort) record_error(p.status, abort, EBD_ERR_TIMEOUT);
        break;
      }
      tc_fence_after();
      // this CTA's vocabulary rows of the chunk: units [u + ulo, u + ulo + 2)
      // of W, i.e. vocabulary indices from p.v_off + (u + ulo) * kUnit
      const int wbase = (u + ulo) * kUnit;
      const int valid = min(min(2, nu - ulo) * kUnit, p.V - wbase);
      const int vbase = p.v_off + wbase;
      const uint32_t taddr0 = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                              static_cast<uint32_t>(buf * p.acc_stride);
      auto rel = [&]() { release(buf); };
      const bool released = epilogue_buffer(taddr0, wg, p.nwg, p.n_pad, sTw, lanev, et, bar_id,
                                            vbase, valid, st_m, st_s, st_t, st_l2, st_i, rel);
      if (!released) release(buf);  // no slice of this chunk for this warpgroup
    }
    if (ok && active) {
      // the rows of this warpgroup's slices (its threads updated them last):
      // this CTA's partial goes to column `col` of its group's rows, and
      // neutral states to the columns [grp_cols, ncols) that no CTA of the
      // group owns
      for (int r = et; r < rows_g; r += 128) {
        if (((r >> 5) % p.nwg) != wg) continue;
        if (!in_bounds(rbase + r, p.part_rows, p.status) || !in_bounds(col, p.ncols, p.status)) continue;
        const size_t o = static_cast<size_t>(rbase + r) * p.ncols + col;
        p.part_f[o] = make_float4(st_m[r], st_s[r], st_t[r], st_l2[r]);
        p.part_i[o] = st_i[r];
        for (int jc = p.grp_cols + col; jc < p.ncols; jc += p.grp_cols) {  // neutral states
          p.part_f[o - col + jc] = make_float4(-INFINITY, 0.f, 0.f, -INFINITY);
          p.part_i[o - col + jc] = INT_MAX;
        }
      }
    }
  }

  __syncthreads();
  // the peer's MMAs, copies and arrivals that target this CTA are over
  if (PAIR) cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    if (PAIR)
      tmem_dealloc_pair(tmem_base, p.tmem_cols);
    else
      tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

// CTAs of the unpaired launch (one per SM at most): the vocabulary units
// spread over the fewest CTAs that take at most one unit more each than an
// even split over every SM, as long as that keeps 90 % of the SMs.  Fewer
// concurrent W streams draw more of the HBM bandwidth: LLaDA-8B (1976 units)
// on 152 CTAs of 13 units 157.9 us, on 142 CTAs of at most 14 154.7 us;
// 148 CTAs 158.9 us, 140 CTAs (at most 15 units) 166.6 us.
int lm_grid(int num_sms, int n_units) {
  if (num_sms < 1) num_sms = 1;
  if (n_units <= num_sms) return n_units < 1 ? 1 : n_units;
  const int per = (n_units + num_sms - 1) / num_sms + 1;
  const int g = (n_units + per - 1) / per;
  return 10 * g >= 9 * num_sms ? g : num_sms;
}

// CTAs of the paired launch: one pair per two SMs, at most one per 4-unit
// chunk of the vocabulary
int lm_pair_grid(int num_sms, int n_units) {
  int np = num_sms / 2;
  const int chunks = (n_units + 3) / 4;
  if (np > chunks) np = chunks;
  if (np < 1) np = 1;
  return 2 * np;
}

void lm_plan(LmParams& p, int rows, int V, int d, int num_sms, bool pair) {
  p.V = V;
  p.d = d;
  p.rows = rows;
  p.pair = pair ? 1 : 0;
  // Paired launches of more than 432 rows split the rows into two groups of
  // at most 256, each served by half the pairs over the whole vocabulary:
  // every CTA's accumulator then fits twice in TMEM, so the epilogue of one
  // chunk overlaps the MMAs of the next, and LLaDA-8B's 494 chunks split
  // evenly over 38 pairs (6.5 per pair otherwise), at the cost of each W tile
  // being read by two pairs (the second read from L2) and ~33 % more operand
  // bytes per flop.  Measured (LM head): 512 rows 401 -> 378 us, 1024 rows
  // 796 -> 751 us, 4096 rows 3188 -> 3021 us; but Dream-7B's 390 rows (groups
  // of 208) 361 -> 396 us, hence the threshold.
  p.rgroups = pair && rows > 432 ? (rows + 255) / 256 : 1;
  if (const char* env = getenv("EBD_LM_RGROUPS")) p.rgroups = pair && atoi(env) > 1 ? (rows + 255) / 256 : 1;
  p.nsub = p.rgroups > 1 ? 1 : (rows + 255) / 256;
  if (p.nsub < 1) p.nsub = 1;
  p.nb = p.rgroups > 1 ? ((rows + p.rgroups - 1) / p.rgroups + 15) / 16 * 16
                       : ((rows + p.nsub - 1) / p.nsub + 15) / 16 * 16;
  if (p.nb < 16) p.nb = 16;
  p.n_pad = p.nb * p.nsub;
  p.acc_stride = (p.n_pad + 31) / 32 * 32;
  p.nbuf = (2 * p.acc_stride <= 512) ? 2 : 1;
  int cols = p.nbuf * p.acc_stride;
  int tc = 32;
  while (tc < cols) tc <<= 1;
  p.tmem_cols = tc;
  p.n_units = (V + kUnit - 1) / kUnit;
  if (pair) {  // 4 units per accumulator; the pairs split evenly over the row groups
    p.nwork = lm_pair_grid(num_sms / p.rgroups, p.n_units) / 2;
    p.grid = 2 * p.nwork * p.rgroups;
    p.grp_cols = 2 * p.nwork;
  } else {
    p.grid = lm_grid(num_sms, p.n_units);
    p.nwork = p.grid;
    p.grp_cols = p.grid;
  }
  p.ncols = p.grp_cols;  // partial states per row (a caller may raise it: neutral states)
  // a second epilogue warpgroup (and its transpose buffer) only pays where
  // the epilogue is exposed, i.e. with a single accumulator buffer; with two,
  // one warpgroup keeps up with the MMAs and its buffer is worth more as
  // pipeline stages (measured with 128-row tiles: 256 rows 270.7 -> 247.2 us)
  p.nwg = p.nbuf == 1 ? 2 : 1;
  if (const char* env = getenv("EBD_LM_NWG")) p.nwg = atoi(env) == 2 ? 2 : 1;
  const uint32_t st_bytes = static_cast<uint32_t>(p.n_pad) * 20u;
  const uint32_t tail = kTBytes * static_cast<uint32_t>(p.nwg) + ((st_bytes + 7) / 8 * 8) +
                        (2 * 8 + 6) * 8 + 16;
  const uint32_t budget = 232448u - 1024u - tail;
  p.nkb = (d + 63) / 64;
  // hidden bytes per k-box in one CTA: all rows, or half of them in a pair
  const uint32_t b_box = static_cast<uint32_t>(pair ? p.n_pad / 2 : p.n_pad) * 128u;
  // k-boxes (64 columns each) per pipeline stage, while keeping at least two
  // stages in flight.  Unpaired (few rows, HBM bound): up to 5, for longer
  // contiguous runs of each W row per request.  Paired: about 512 / N, so
  // that a stage's MMAs keep the tensor cores busy for about as long at any
  // N: measured at 128 rows 4 k-boxes x 2 stages 172 us, 2 x 4 197 us; 256
  // rows 2 x 3 214 us, 3 x 2 223 us, 1 x 6 272 us; 390 rows 1 x 4 360 us,
  // 2 x 2 367 us.  Smaller stages cost more in hand-offs than their depth
  // gains (one k-box per stage in separate W and hidden-row rings: 256 rows
  // 434 us).
  int kbs = pair ? 512 / p.n_pad : 5;
  if (const char* env = getenv("EBD_LM_KBS")) kbs = atoi(env);
  if (kbs < 1) kbs = 1;
  if (kbs > 5) kbs = 5;
  if (kbs > p.nkb) kbs = p.nkb;
  while (kbs > 1 && budget / (static_cast<uint32_t>(kbs) * (kATile + b_box)) < 2) --kbs;
  p.kbs = kbs;
  p.nks = (p.nkb + kbs - 1) / kbs;
  const uint32_t stage = static_cast<uint32_t>(kbs) * (kATile + b_box);
  int stages = static_cast<int>(budget / stage);
  if (stages > 8) stages = 8;
  p.stages = stages;
  p.off_a = 0;
  p.off_b = p.off_a + static_cast<uint32_t>(stages) * kbs * kATile;
  p.off_t = p.off_b + static_cast<uint32_t>(stages) * kbs * b_box;
  p.off_st = p.off_t + kTBytes * static_cast<uint32_t>(p.nwg);
  p.off_bar = (p.off_st + st_bytes + 7) / 8 * 8;
  p.smem_bytes = p.off_bar + static_cast<uint32_t>(2 * stages + 6) * 8u + 16u + 1024u;
}

// Tiled copy of W: out[((u * nkb + k) * 64 + r) * 64 + c] = W[64u + r][64k + c]
__global__ void __launch_bounds__(256) pack_lm_kernel(const uint4* __restrict__ w,
                                                      uint4* __restrict__ out, int V, int d,
                                                      int nkb, long long n_vec) {
  const long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n_vec) return;
  const int c8 = static_cast<int>(i & 7);          // 8 bf16 per 16-byte vector
  const long long row = i >> 3;                    // packed row (64 columns)
  const int r = static_cast<int>(row & 63);
  const long long tile = row >> 6;
  const int kb = static_cast<int>(tile % nkb);
  const long long u = tile / nkb;
  const long long v = u * 64 + r;
  const int col = kb * 64 + c8 * 8;
  uint4 val = make_uint4(0u, 0u, 0u, 0u);
  if (v < V && col < d) {
    if (col + 8 <= d && (d % 8) == 0) {
      val = w[(v * d + col) / 8];
    } else {
      const __nv_bfloat16* ws = reinterpret_cast<const __nv_bfloat16*>(w);
      __nv_bfloat16 t[8];
      for (int e = 0; e < 8; ++e)
        t[e] = (col + e < d) ? ws[v * d + col + e] : __float2bfloat16(0.f);
      val = *reinterpret_cast<uint4*>(t);
    }
  }
  out[i] = val;
}

cudaError_t launch_pack_lm(const __nv_bfloat16* w, __nv_bfloat16* out, int V, int d,
                           cudaStream_t st) {
  const int nkb = (d + 63) / 64;
  const long long units = (V + 63) / 64;
  const long long n_vec = units * nkb * 64 * 8;
  const long long blocks = (n_vec + 255) / 256;
  pack_lm_kernel<<<static_cast<unsigned>(blocks), 256, 0, st>>>(
      reinterpret_cast<const uint4*>(w), reinterpret_cast<uint4*>(out), V, d, nkb, n_vec);
  return cudaGetLastError();
}

cudaError_t lm_configure() {
  const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(lm_stats_kernel<true, true>, a, 232448)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(lm_stats_kernel<true, false>, a, 232448)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(lm_stats_kernel<false, true>, a, 232448)) != cudaSuccess) return e;
  return cudaFuncSetAttribute(lm_stats_kernel<false, false>, a, 232448);
}

cudaError_t launch_lm_stats(const CUtensorMap& tmap_w, const CUtensorMap& tmap_h,
                            const LmParams& p, cudaStream_t st) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(p.grid, 1, 1);
  cfg.blockDim = dim3(kLmThreads, 1, 1);
  cfg.dynamicSmemBytes = p.smem_bytes;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (p.pair) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 2;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  if (p.pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  if (p.pair)
    return p.packed ? cudaLaunchKernelEx(&cfg, lm_stats_kernel<true, true>, tmap_w, tmap_h, p)
                    : cudaLaunchKernelEx(&cfg, lm_stats_kernel<true, false>, tmap_w, tmap_h, p);
  return p.packed ? cudaLaunchKernelEx(&cfg, lm_stats_kernel<false, true>, tmap_w, tmap_h, p)
                  : cudaLaunchKernelEx(&cfg, lm_stats_kernel<false, false>, tmap_w, tmap_h, p);
}

}  // namespace ebd
