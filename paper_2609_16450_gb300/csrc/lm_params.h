// Launch parameters of the LM-head kernel (k_lmhead.cu), shared with the
// host code that plans and launches it.
#pragma once
#include <cuda_runtime.h>
#include <cstdint>

namespace ebd {

struct LmParams {
  int V, d;                 // vocabulary rows of this launch's W, hidden size
  int v_off;                // vocabulary index of W's first row (a shard's offset; 0 otherwise)
  int row0, rows;           // rows [row0, row0 + rows) of this launch
  int nb, nsub, n_pad;      // MMA N per sub-tile, sub-tiles, padded N = nb * nsub
  int n_units;              // ceil(V / 64)
  int grid;                 // CTAs (each writes one partial per row)
  int nkb;                  // ceil(d / 64) k-blocks of 64 columns
  int kbs, nks;             // k-blocks per pipeline stage, stages per vocabulary chunk
  int packed;               // W is tiled: tile (unit, k-block) at row (unit*nkb + kb)*64
  int stages, nbuf, acc_stride, tmem_cols;
  int nwg;                  // epilogue warpgroups in use (2 with a single accumulator buffer)
  int pair;                 // CTA pairs (clusters of 2) running cta_group::2 MMAs, M = 256
  int nwork;                // owners of vocabulary ranges per row group: CTAs, or pairs
  int rgroups;              // row groups (paired launches of more than 256 rows: 2), each
                            // of nb rows, served by its own nwork owners
  int grp_cols;             // CTAs per row group (the partial columns a row gets here)
  int ncols;                // partial states per row written (>= grid; extra ones neutral)
  int part_rows;            // rows the partial buffers hold
  uint32_t off_a, off_b, off_t, off_st, off_bar, smem_bytes;
  float4* part_f;           // [R][grid] (max, sum exp, sum exp*(l-max), second logit)
  int* part_i;              // [R][grid] argmax
  int* status;
  uint64_t limit_ns;
  int force_timeout;
  int pdl;                  // a programmatic dependent of the kernel before it, which
                            // copies the hidden rows in: W loads start before the wait
};

}  // namespace ebd
