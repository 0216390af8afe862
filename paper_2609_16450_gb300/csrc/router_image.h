// Device image of the router weights, laid out for the decision kernel.
//
// The LBS encoder is split over the 8 CTAs of a cluster by output features
// (rank r owns QKV features [48r, 48r+48), projection/combine outputs
// [16r, 16r+16) and FFN hidden units [32r, 32r+32)).  Each rank's matrices
// are stored transposed ([in][out], bf16) in one contiguous block, so a CTA
// loads everything it needs with one bulk copy; vectors are fp32.
#pragma once

namespace ebd {
namespace rimg {

constexpr int kRanks = 8;
constexpr int kQkvSlice = 48, kOutSlice = 16, kFf1Slice = 32, kCombSlice = 16;
constexpr int kPosRows = 64;  // E_pos rows a window can use

// ---- LBS weights of one rank, bf16 elements
constexpr int W_ENT2 = 0;         // [64][64]   ent2 (full)
constexpr int W_COMB = 4096;      // [128][16]  combine slice
constexpr int W_POS = 6144;       // [64][16]   E_pos slice
constexpr int W_LAYER0 = 7168;    // two layers of W_LAYER_STRIDE
constexpr int W_LAYER_STRIDE = 16384;
constexpr int WL_QKV = 0;         // [128][48]  QKV feature slice
constexpr int WL_OUT = 6144;      // [128][16]  output projection slice
constexpr int WL_FF1 = 8192;      // [128][32]  FFN first linear, hidden slice
constexpr int WL_FF2 = 12288;     // [32][128]  FFN second linear, rows of the hidden slice
constexpr int LBS_W_ELEMS = W_LAYER0 + 2 * W_LAYER_STRIDE;  // 39936

// The LBS matrices above except E_pos are stored with their 16-byte chunks
// permuted within each row: element (k, c) of a [K][ld] matrix sits at
// k * ld + swz_col(k, c, ld).  ldmatrix reads 8 consecutive rows of one
// 8-column chunk as an mma B fragment; the XOR places those 8 row segments in
// 8 distinct 16-byte bank groups for ld = 16, 32, 48, 64 and 128 (without it,
// rows of 128 or 256 bytes put all 8 in one group).  K is a multiple of 16,
// and the mask depends only on the low 3 bits of k.
__host__ __device__ constexpr int swz_mask(int k, int ld) {
  return ld >= 64 ? (k & 7) : ld == 32 ? ((k >> 1) & 3) : ((k >> 2) & 1);
}
__host__ __device__ constexpr int swz_col(int k, int c, int ld) {
  return (((c >> 3) ^ swz_mask(k, ld)) << 3) | (c & 7);
}

// ---- LPS weights (one copy), bf16, transposed [in][out] with each row padded
// by 8 elements so that 8 consecutive rows hit distinct banks when ldmatrix
// reads them as mma B fragments
constexpr int PL_QKV = 0;         // [32][104]
constexpr int PL_OUT = 3328;      // [32][40]
constexpr int PL_FF1 = 4608;      // [32][72]
constexpr int PL_FF2 = 6912;      // [64][40]
constexpr int PL_STRIDE = 9472;
constexpr int PL_LDQKV = 104, PL_LDOUT = 40, PL_LDFF1 = 72, PL_LDFF2 = 40;
constexpr int LPS_W_ELEMS = 2 * PL_STRIDE;

// ---- fp32 vectors of one rank
constexpr int V_ENT1W = 0, V_ENT1B = 64, V_ENT2B = 128, V_ENTLNG = 192, V_ENTLNB = 256;
constexpr int V_TOKB = 320, V_HEADW = 384, V_HEADB = 512, V_COMBB = 516;
constexpr int V_LAYER0 = 544, V_LAYER_STRIDE = 624;
constexpr int VL_QKVB = 0, VL_OUTB = 48, VL_FF1B = 64, VL_FF2B = 96;
constexpr int VL_LN1G = 112, VL_LN1B = 240, VL_LN2G = 368, VL_LN2B = 496;
constexpr int V_LPS = 1792;
constexpr int VP_INT = 0, VP_INB = 160, VP_INLNG = 192, VP_INLNB = 224, VP_HEADW = 256;
constexpr int VP_HEADB = 288, VP_LAYER0 = 292, VP_LAYER_STRIDE = 352;
constexpr int VPL_LN1G = 0, VPL_LN1B = 32, VPL_QKVB = 64, VPL_OUTB = 160, VPL_LN2G = 192;
constexpr int VPL_LN2B = 224, VPL_FF1B = 256, VPL_FF2B = 320;
constexpr int V_ELEMS = 2800;

static_assert(V_LAYER0 + 2 * V_LAYER_STRIDE <= V_LPS, "vector layout");
static_assert(V_LPS + VP_LAYER0 + 2 * VP_LAYER_STRIDE <= V_ELEMS, "vector layout");
static_assert(LPS_W_ELEMS <= LBS_W_ELEMS, "LPS weights reuse the LBS weight region");
static_assert((LBS_W_ELEMS * 2) % 16 == 0 && (LPS_W_ELEMS * 2) % 16 == 0 &&
                  (V_ELEMS * 4) % 16 == 0,
              "bulk copies move multiples of 16 bytes");

// ---- the one-CTA decision kernel (windows of up to 32 rows).  Its LBS
// products run on the tcgen05 tensor cores with the weights as the A operand:
// every matrix W [out][in] is cut into tiles of 128 output rows x 64 inputs,
// each stored as the K-major, 128-byte-swizzled shared-memory image the MMA
// reads (row m at m * 128 bytes; its 16-byte chunk c at chunk c ^ (m & 7)),
// 16 KB, so that one bulk copy moves one tile into a slot of a ring.  The
// tiles are stored in the order the kernel consumes them; a tile of a
// product with T output tiles and K / 64 input boxes is at chunk t * (K / 64)
// + kb.  Rows beyond a matrix's outputs are zero.
namespace rcta {

constexpr int kChunkElems = 8192;  // bf16 elements per chunk (16 KB)
constexpr int kPosRows = 32;       // E_pos rows a window can use
constexpr int C_ENT = 0;           // ent2: 64 output rows of 128, K = 64
constexpr int C_COMB = 1;          // 2 chunks: combine, 128 outputs, K = 128
constexpr int C_LAYER0 = 3;        // encoder layer l at C_LAYER0 + l * CL_CHUNKS
constexpr int CL_QKV = 0;          // 6 chunks: 384 outputs (3 tiles), K = 128
constexpr int CL_OUT = 6;          // 2 chunks: output projection, K = 128
constexpr int CL_FF1 = 8;          // 4 chunks: 256 hidden units (2 tiles), K = 128
constexpr int CL_FF2 = 12;         // 4 chunks: 128 outputs, K = 256
constexpr int CL_CHUNKS = 16;
constexpr int C_LPS = C_LAYER0 + 2 * CL_CHUNKS;  // the LPS weights (PL_* layout above)
constexpr int LPS_CHUNKS = (LPS_W_ELEMS + kChunkElems - 1) / kChunkElems;
constexpr int kChunks = C_LPS + LPS_CHUNKS;

// element (m, k) of a 128 x 64 tile, in bf16 elements from the tile start
__host__ __device__ constexpr int tile_off(int m, int k) {
  return m * 64 + ((((k >> 3) ^ (m & 7)) << 3) | (k & 7));
}

// fp32 vectors, whole; then E_pos [32][128] as bf16 (S_POS, in floats)
constexpr int S_ENT1W = 0, S_ENT1B = 64, S_ENT2B = 128, S_ENTLNG = 192, S_ENTLNB = 256;
constexpr int S_TOKB = 320, S_COMBB = 384, S_HEADW = 512, S_HEADB = 640;
constexpr int S_LAYER0 = 656, S_LAYER_STRIDE = 1408;
constexpr int SL_QKVB = 0, SL_OUTB = 384, SL_FF1B = 512, SL_FF2B = 768;
constexpr int SL_LN1G = 896, SL_LN1B = 1024, SL_LN2G = 1152, SL_LN2B = 1280;
constexpr int S_LPS = S_LAYER0 + 2 * S_LAYER_STRIDE;  // the LPS vectors (VP_* layout above)
constexpr int S_POS = S_LPS + 1008;
constexpr int S_ELEMS = S_POS + kPosRows * 128 / 2;

static_assert(S_LPS + VP_LAYER0 + 2 * VP_LAYER_STRIDE <= S_POS, "vector layout");
static_assert(S_LAYER0 % 4 == 0 && S_LAYER_STRIDE % 4 == 0 && S_LPS % 4 == 0 &&
                  S_POS % 4 == 0 && (S_ELEMS * 4) % 16 == 0,
              "float4 alignment of LayerNorm vectors, bulk copy size");
static_assert(LPS_CHUNKS == 3, "the LPS weights take three chunks");

}  // namespace rcta

}  // namespace rimg
}  // namespace ebd
