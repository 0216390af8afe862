// Host side of the C ABI declared in include/ebd.h.
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdlib>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "ebd.h"
#include "internal.h"
#include "router_image.h"

namespace {
// An NVTX range around the host side of an entry point (visible in Nsight
// Systems timelines; a no-op when no tool is attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
};
}  // namespace

namespace ebd {
cudaError_t decide_configure();
cudaError_t decide_cta_configure();
cudaError_t attn_configure();
cudaError_t lm_configure();
cudaError_t launch_merge_stats(const float4* part_f, const int* part_i, int rows, int grid,
                               int V, float inv_log_v, float* conf, float* entropy,
                               float* ent_norm, float* gap, int* argmax, int* status,
                               cudaStream_t st, bool pdl = false);
}  // namespace ebd

using namespace ebd;

namespace {

constexpr uint64_t kLimitNs = 1000ull * 1000 * 1000;  // 1 s per device-side wait
constexpr int kMaxSplits = kMaxAttnSplits;

// ------------------------------------------------------------------ router layout
struct TensorDesc {
  std::string name;
  int rows, cols;  // row-major [rows][cols]; vectors have rows = 1
  int kind;        // 0 linear (fan_in), 1 ones, 2 zeros, 3 positional
  int fan_in;
};

std::vector<TensorDesc> router_layout(int d_base, int gen_len) {
  std::vector<TensorDesc> t;
  auto lin = [&](const std::string& n, int o, int i) {
    t.push_back({n + ".w", o, i, 0, i});
    t.push_back({n + ".b", 1, o, 0, i});
  };
  auto ln = [&](const std::string& n, int d) {
    t.push_back({n + ".g", 1, d, 1, 0});
    t.push_back({n + ".b", 1, d, 2, 0});
  };
  lin("lbs.ent1", 64, 1);
  lin("lbs.ent2", 64, 64);
  ln("lbs.ent_ln", 64);
  lin("lbs.tok", 64, d_base);
  lin("lbs.comb", 128, 128);
  t.push_back({"lbs.pos", gen_len, 128, 3, 0});
  for (int l = 0; l < 2; ++l) {
    const std::string p = "lbs.l" + std::to_string(l);
    lin(p + ".qkv", 384, 128);
    lin(p + ".out", 128, 128);
    ln(p + ".ln1", 128);
    lin(p + ".ff1", 256, 128);
    lin(p + ".ff2", 128, 256);
    ln(p + ".ln2", 128);
  }
  lin("lbs.head", 1, 128);
  lin("lps.in", 32, 5);
  ln("lps.in_ln", 32);
  for (int l = 0; l < 2; ++l) {
    const std::string p = "lps.l" + std::to_string(l);
    ln(p + ".ln1", 32);
    lin(p + ".qkv", 96, 32);
    lin(p + ".out", 32, 32);
    ln(p + ".ln2", 32);
    lin(p + ".ff1", 64, 32);
    lin(p + ".ff2", 32, 64);
  }
  lin("lps.head", 1, 32);
  return t;
}

size_t layout_count(const std::vector<TensorDesc>& t) {
  size_t n = 0;
  for (const auto& x : t) n += static_cast<size_t>(x.rows) * x.cols;
  return n;
}

// SplitMix64 output function (Steele, Lea & Flood 2014)
inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return static_cast<uint16_t>(u >> 16);
}
inline float bf16_to_f32(uint16_t b) {
  uint32_t u = static_cast<uint32_t>(b) << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

void router_init(uint64_t seed, const std::vector<TensorDesc>& layout, uint16_t* out) {
  const uint64_t G = 0x9E3779B97F4A7C15ull;
  size_t off = 0;
  for (size_t ti = 0; ti < layout.size(); ++ti) {
    const TensorDesc& t = layout[ti];
    const size_t n = static_cast<size_t>(t.rows) * t.cols;
    if (t.kind == 1) {
      for (size_t i = 0; i < n; ++i) out[off + i] = 0x3F80;
    } else if (t.kind == 2) {
      for (size_t i = 0; i < n; ++i) out[off + i] = 0;
    } else {
      const float bound = t.kind == 0 ? 1.0f / std::sqrt(static_cast<float>(t.fan_in))
                                      : 0.02f * std::sqrt(3.0f);
      const uint64_t key = mix64(seed ^ ((static_cast<uint64_t>(ti) + 1) * G));
      for (size_t i = 0; i < n; ++i) {
        const uint64_t z = mix64(key + (static_cast<uint64_t>(i) + 1) * G);
        const float u = static_cast<float>(z >> 40) * (1.0f / 16777216.0f);
        const float v = 2.0f * u - 1.0f;
        out[off + i] = f32_to_bf16_rne(v * bound);
      }
    }
    off += n;
  }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

bool encode_bf16(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                 const uint64_t* strides_bytes, const uint32_t* box) {
  auto fn = get_encode();
  if (fn == nullptr) return false;
  cuuint64_t gd[5], gs[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) {
    gd[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
  }
  for (int i = 0; i < rank - 1; ++i) gs[i] = strides_bytes[i];
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, static_cast<cuuint32_t>(rank),
                  const_cast<void*>(base), gd, gs, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Tensor map of W_lm in boxes of 64 columns by 64 rows: row-major [V][d], or
// the packed layout ([unit][k-box][64 rows][64 columns], ebd_pack_lm_head).
// For CTA pairs (pair_kbs > 0 k-boxes per stage) the packed layout is read as
// a 4-D tensor (column, row, unit, k-box) in boxes of two units by pair_kbs
// k-boxes: one box is a CTA's 128 W rows of a whole pipeline stage.
bool encode_w_lm(CUtensorMap* m, const void* w, int V, int d, bool packed, int pair_kbs) {
  const uint64_t units = (static_cast<uint64_t>(V) + kUnit - 1) / kUnit;
  const uint64_t nkb = (static_cast<uint64_t>(d) + 63) / 64;
  if (packed && pair_kbs > 0) {
    const uint64_t dims[4] = {64ull, 64ull, units, nkb};
    const uint64_t str[3] = {128ull, nkb * 64 * 128, 64 * 128};
    const uint32_t box[4] = {64, 64, 2, static_cast<uint32_t>(pair_kbs)};
    return encode_bf16(m, w, 4, dims, str, box);
  }
  const uint64_t dims[2] = {packed ? 64ull : static_cast<uint64_t>(d),
                            packed ? units * nkb * 64 : static_cast<uint64_t>(V)};
  const uint64_t str[1] = {packed ? 128ull : static_cast<uint64_t>(d) * 2};
  const uint32_t box[2] = {64, 64};
  return encode_bf16(m, w, 2, dims, str, box);
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Event record that also executes when the stream is being captured into a
// CUDA graph (an external event-record node rather than a dependency edge).
cudaError_t record(cudaEvent_t ev, cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(st, &cs);
  if (e != cudaSuccess) return e;
  if (cs == cudaStreamCaptureStatusActive)
    return cudaEventRecordWithFlags(ev, st, cudaEventRecordExternal);
  return cudaEventRecord(ev, st);
}

}  // namespace

struct ebd_handle {
  ebd_config cfg{};
  int device = 0, num_sms = 0;
  std::string err;
  std::vector<TensorDesc> layout;
  std::vector<uint16_t> h_blob;
  uint16_t* d_blob = nullptr;
  uint8_t* d_image = nullptr;
  RouterImage img{};
  float* d_tok = nullptr;
  const uint16_t* w_emb = nullptr;
  float4* part_f = nullptr;
  int* part_i = nullptr;
  int grid_lm = 0;       // LM-head partial states per row
  int lm_ctas = 0;       // CTAs of the last LM-head launch (one SM each)
  int lm_units = 0;      // 64-row vocabulary units
  float* attn_part = nullptr;
  float* attn_part_ml = nullptr;
  int* tickets = nullptr;
  int attn_splits = 1, attn_max_qtiles = 1;
  int attn_tc = 1;         // window attention on tcgen05 (else the mma.sync kernel)
  int* d_status = nullptr;
  uint8_t* staging = nullptr;
  size_t staging_bytes = 0;
  // the grid-wide decision (max_window > kMaxWindow)
  float* d_seqw = nullptr;   // SeqWeights image
  SeqWeights seqw{};
  uint8_t* seq_scratch = nullptr;
  SeqParams seqp{};          // scratch pointers, filled at create
  cudaEvent_t ev[4] = {nullptr, nullptr, nullptr, nullptr};
  int profile = 0;
  int prof_mode = 0, prof_attn = 0;  // what the last ebd_step recorded
  // ebd_step_host: the attention's inputs on a copy engine (set up with the handle)
  int copy_route = -1;               // -1 not set up yet, 0 unavailable, 1 ready
  cudaStream_t s_copy = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  unsigned* d_ready = nullptr;
  unsigned ticket = 0;
};

namespace {

typedef CUresult (*WriteValue32Fn)(CUstream, CUdeviceptr, cuuint32_t, unsigned int);
WriteValue32Fn get_write_value() {
  static WriteValue32Fn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuStreamWriteValue32", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<WriteValue32Fn>(ptr);
  });
  return fn;
}

// The copy stream, its two events and the ticket word; false where the
// driver offers no stream write (the inputs then go with the others).
bool copy_route_ready(ebd_handle* h) {
  if (h->copy_route >= 0) return h->copy_route == 1;
  h->copy_route = 0;
  if (get_write_value() == nullptr) return false;
  if (cudaStreamCreateWithFlags(&h->s_copy, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming) != cudaSuccess ||
      cudaMalloc(&h->d_ready, sizeof(unsigned)) != cudaSuccess ||
      cudaMemsetAsync(h->d_ready, 0, sizeof(unsigned), h->s_copy) != cudaSuccess ||
      cudaStreamSynchronize(h->s_copy) != cudaSuccess) {
    (void)cudaGetLastError();
    return false;
  }
  h->copy_route = 1;
  return true;
}

ebd_status fail(ebd_handle* h, ebd_status code, const std::string& msg) {
  if (h) h->err = msg;
  return code;
}
ebd_status cuda_fail(ebd_handle* h, cudaError_t e, const char* what) {
  return fail(h, EBD_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

ebd_status validate_config(const ebd_config* c, std::string& why) {
  auto bad = [&](const char* m) {
    why = m;
    return EBD_ERR_UNSUPPORTED;
  };
  if (c->d_model <= 0 || c->d_model % 8) return bad("d_model must be a positive multiple of 8");
  if (c->d_base <= 0 || c->d_base % 8) return bad("d_base must be a positive multiple of 8");
  if (c->vocab < 2) return bad("vocab must be >= 2");
  if (c->head_dim != 64 && c->head_dim != 128) return bad("head_dim must be 64 or 128");
  if (c->n_heads_kv <= 0 || c->n_heads_q <= 0 || c->n_heads_q % c->n_heads_kv)
    return bad("n_heads_q must be a positive multiple of n_heads_kv");
  if (c->max_batch <= 0 || c->max_batch > 65535) return bad("max_batch out of range");
  if (c->max_window <= 0 || c->max_window > kMaxSeqRows) return bad("max_window must be 1..512");
  if (c->max_rows <= 0 || c->max_rows > 4096) return bad("max_rows must be 1..4096");
  if (c->max_prefix < 0) return bad("max_prefix must be >= 0");
  if (c->gen_len < c->max_window) return bad("gen_len must be >= max_window");
  if (c->g_max < 0 || c->l_min < 0 || c->l_b < 0) return bad("g_max, l_min, l_b must be >= 0");
  if (!(c->tau == c->tau) || !(c->tau_psi == c->tau_psi)) return bad("tau/tau_psi is NaN");
  if (c->decode_mode < EBD_DECODE_EB || c->decode_mode > EBD_DECODE_TOPM)
    return bad("decode_mode must be EBD_DECODE_EB, _THRESHOLD or _TOPM");
  if (c->decode_mode == EBD_DECODE_TOPM && c->top_m < 1) return bad("top_m must be >= 1");
  return EBD_OK;
}

ebd_status check_device(ebd_handle* h) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaGetDevice");
  if (dev != h->device) return fail(h, EBD_ERR_INVALID_ARG, "current device differs from the handle's");
  return EBD_OK;
}

// fp32 image of the router weights for the grid-wide decision: matrices
// [in][out], vectors as they are (SeqWeights).
ebd_status upload_seq_weights(ebd_handle* h) {
  // element (r, c) of a blob tensor, its offset resolved once per name
  std::string last;
  size_t last_off = 0, last_cols = 0;
  auto atf = [&](const std::string& name, int r, int c) -> float {
    if (name != last) {
      size_t off = 0;
      bool found = false;
      for (const auto& t : h->layout) {
        if (t.name == name) {
          last_cols = static_cast<size_t>(t.cols);
          found = true;
          break;
        }
        off += static_cast<size_t>(t.rows) * t.cols;
      }
      last = name;
      last_off = found ? off : 0;
    }
    return bf16_to_f32(h->h_blob[last_off + static_cast<size_t>(r) * last_cols + c]);
  };
  SeqWeights& o = h->seqw;
  int n = 0;
  auto take = [&](int count) {
    const int at = n;
    n += (count + 3) / 4 * 4;
    return at;
  };
  const int L = h->cfg.gen_len;
  o.ent1_w = take(64); o.ent1_b = take(64); o.ent2_t = take(64 * 64); o.ent2_b = take(64);
  o.entln_g = take(64); o.entln_b = take(64); o.tok_b = take(64);
  o.comb_t = take(128 * 128); o.comb_b = take(128); o.pos = take(L * 128);
  for (int l = 0; l < 2; ++l) {
    SeqLayer& q = o.l[l];
    q.qkv_t = take(128 * 384); q.qkv_b = take(384); q.out_t = take(128 * 128); q.out_b = take(128);
    q.ln1_g = take(128); q.ln1_b = take(128); q.ff1_t = take(128 * 256); q.ff1_b = take(256);
    q.ff2_t = take(256 * 128); q.ff2_b = take(128); q.ln2_g = take(128); q.ln2_b = take(128);
  }
  o.head_w = take(128); o.head_b = take(1);
  o.in_t = take(5 * 32); o.in_b = take(32); o.inln_g = take(32); o.inln_b = take(32);
  for (int l = 0; l < 2; ++l) {
    SeqBlock& q = o.p[l];
    q.ln1_g = take(32); q.ln1_b = take(32); q.qkv_t = take(32 * 96); q.qkv_b = take(96);
    q.out_t = take(32 * 32); q.out_b = take(32); q.ln2_g = take(32); q.ln2_b = take(32);
    q.ff1_t = take(32 * 64); q.ff1_b = take(64); q.ff2_t = take(64 * 32); q.ff2_b = take(32);
  }
  o.phead_w = take(32); o.phead_b = take(1);
  o.total = n;
  std::vector<float> w(static_cast<size_t>(n), 0.f);
  // [in][out] copy of a [out][in] matrix, and a vector
  auto mat = [&](int at, const std::string& name, int nin, int nout) {
    for (int k = 0; k < nin; ++k)
      for (int c = 0; c < nout; ++c) w[at + static_cast<size_t>(k) * nout + c] = atf(name, c, k);
  };
  auto vec = [&](int at, const std::string& name, int count) {
    for (int c = 0; c < count; ++c) w[at + c] = atf(name, 0, c);
  };
  for (int c = 0; c < 64; ++c) w[o.ent1_w + c] = atf("lbs.ent1.w", c, 0);
  vec(o.ent1_b, "lbs.ent1.b", 64);
  mat(o.ent2_t, "lbs.ent2.w", 64, 64);
  vec(o.ent2_b, "lbs.ent2.b", 64);
  vec(o.entln_g, "lbs.ent_ln.g", 64);
  vec(o.entln_b, "lbs.ent_ln.b", 64);
  vec(o.tok_b, "lbs.tok.b", 64);
  mat(o.comb_t, "lbs.comb.w", 128, 128);
  vec(o.comb_b, "lbs.comb.b", 128);
  for (int j = 0; j < L; ++j)
    for (int c = 0; c < 128; ++c) w[o.pos + static_cast<size_t>(j) * 128 + c] = atf("lbs.pos", j, c);
  for (int l = 0; l < 2; ++l) {
    const std::string pre = "lbs.l" + std::to_string(l);
    const SeqLayer& q = o.l[l];
    mat(q.qkv_t, pre + ".qkv.w", 128, 384); vec(q.qkv_b, pre + ".qkv.b", 384);
    mat(q.out_t, pre + ".out.w", 128, 128); vec(q.out_b, pre + ".out.b", 128);
    vec(q.ln1_g, pre + ".ln1.g", 128); vec(q.ln1_b, pre + ".ln1.b", 128);
    mat(q.ff1_t, pre + ".ff1.w", 128, 256); vec(q.ff1_b, pre + ".ff1.b", 256);
    mat(q.ff2_t, pre + ".ff2.w", 256, 128); vec(q.ff2_b, pre + ".ff2.b", 128);
    vec(q.ln2_g, pre + ".ln2.g", 128); vec(q.ln2_b, pre + ".ln2.b", 128);
  }
  vec(o.head_w, "lbs.head.w", 128);
  vec(o.head_b, "lbs.head.b", 1);
  mat(o.in_t, "lps.in.w", 5, 32);
  vec(o.in_b, "lps.in.b", 32);
  vec(o.inln_g, "lps.in_ln.g", 32);
  vec(o.inln_b, "lps.in_ln.b", 32);
  for (int l = 0; l < 2; ++l) {
    const std::string pre = "lps.l" + std::to_string(l);
    const SeqBlock& q = o.p[l];
    vec(q.ln1_g, pre + ".ln1.g", 32); vec(q.ln1_b, pre + ".ln1.b", 32);
    mat(q.qkv_t, pre + ".qkv.w", 32, 96); vec(q.qkv_b, pre + ".qkv.b", 96);
    mat(q.out_t, pre + ".out.w", 32, 32); vec(q.out_b, pre + ".out.b", 32);
    vec(q.ln2_g, pre + ".ln2.g", 32); vec(q.ln2_b, pre + ".ln2.b", 32);
    mat(q.ff1_t, pre + ".ff1.w", 32, 64); vec(q.ff1_b, pre + ".ff1.b", 64);
    mat(q.ff2_t, pre + ".ff2.w", 64, 32); vec(q.ff2_b, pre + ".ff2.b", 32);
  }
  vec(o.phead_w, "lps.head.w", 32);
  vec(o.phead_b, "lps.head.b", 1);
  if (h->d_seqw == nullptr) {
    cudaError_t e = cudaMalloc(&h->d_seqw, w.size() * sizeof(float));
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMalloc(router fp32 image)");
  }
  cudaError_t e = cudaMemcpy(h->d_seqw, w.data(), w.size() * sizeof(float), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemcpy(router fp32 image)");
  return EBD_OK;
}

// Builds the decision kernel's weight image (router_image.h) from the blob.
ebd_status upload_router(ebd_handle* h) {
  using namespace rimg;
  const auto& L = h->layout;
  std::vector<size_t> off(L.size());
  {
    size_t o = 0;
    for (size_t i = 0; i < L.size(); ++i) {
      off[i] = o;
      o += static_cast<size_t>(L[i].rows) * L[i].cols;
    }
  }
  auto T = [&](const std::string& n) -> const TensorDesc& {
    for (size_t i = 0; i < L.size(); ++i)
      if (L[i].name == n) return L[i];
    return L[0];
  };
  auto idx = [&](const std::string& n) -> size_t {
    for (size_t i = 0; i < L.size(); ++i)
      if (L[i].name == n) return i;
    return 0;
  };
  // element (r, c) of tensor n as bf16 bits / float
  auto at = [&](const std::string& n, int r, int c) -> uint16_t {
    const size_t i = idx(n);
    return h->h_blob[off[i] + static_cast<size_t>(r) * L[i].cols + c];
  };
  auto atf = [&](const std::string& n, int r, int c) { return bf16_to_f32(at(n, r, c)); };
  (void)T;
  std::vector<uint16_t> lbs(static_cast<size_t>(kRanks) * LBS_W_ELEMS, 0);
  std::vector<uint16_t> lps(LPS_W_ELEMS, 0);
  std::vector<float> vec(static_cast<size_t>(kRanks) * V_ELEMS, 0.f);
  const int gen_len = h->cfg.gen_len;
  for (int r = 0; r < kRanks; ++r) {
    uint16_t* w = lbs.data() + static_cast<size_t>(r) * LBS_W_ELEMS;
    float* v = vec.data() + static_cast<size_t>(r) * V_ELEMS;
    for (int k = 0; k < 64; ++k)
      for (int o = 0; o < 64; ++o) w[W_ENT2 + k * 64 + swz_col(k, o, 64)] = at("lbs.ent2.w", o, k);
    for (int k = 0; k < 128; ++k)
      for (int o = 0; o < kCombSlice; ++o)
        w[W_COMB + k * kCombSlice + swz_col(k, o, kCombSlice)] = at("lbs.comb.w", kCombSlice * r + o, k);
    for (int j = 0; j < kPosRows; ++j)
      for (int o = 0; o < kCombSlice; ++o)
        w[W_POS + j * kCombSlice + o] = j < gen_len ? at("lbs.pos", j, kCombSlice * r + o) : 0;
    for (int l = 0; l < 2; ++l) {
      const std::string pre = "lbs.l" + std::to_string(l);
      uint16_t* wl = w + W_LAYER0 + l * W_LAYER_STRIDE;
      float* vl = v + V_LAYER0 + l * V_LAYER_STRIDE;
      for (int k = 0; k < 128; ++k) {
        for (int o = 0; o < kQkvSlice; ++o)
          wl[WL_QKV + k * kQkvSlice + swz_col(k, o, kQkvSlice)] = at(pre + ".qkv.w", kQkvSlice * r + o, k);
        for (int o = 0; o < kOutSlice; ++o)
          wl[WL_OUT + k * kOutSlice + swz_col(k, o, kOutSlice)] = at(pre + ".out.w", kOutSlice * r + o, k);
        for (int o = 0; o < kFf1Slice; ++o)
          wl[WL_FF1 + k * kFf1Slice + swz_col(k, o, kFf1Slice)] = at(pre + ".ff1.w", kFf1Slice * r + o, k);
      }
      for (int hh = 0; hh < kFf1Slice; ++hh)
        for (int o = 0; o < 128; ++o)
          wl[WL_FF2 + hh * 128 + swz_col(hh, o, 128)] = at(pre + ".ff2.w", o, kFf1Slice * r + hh);
      for (int o = 0; o < kQkvSlice; ++o) vl[VL_QKVB + o] = atf(pre + ".qkv.b", 0, kQkvSlice * r + o);
      for (int o = 0; o < kOutSlice; ++o) vl[VL_OUTB + o] = atf(pre + ".out.b", 0, kOutSlice * r + o);
      for (int o = 0; o < kFf1Slice; ++o) vl[VL_FF1B + o] = atf(pre + ".ff1.b", 0, kFf1Slice * r + o);
      for (int o = 0; o < kOutSlice; ++o) vl[VL_FF2B + o] = atf(pre + ".ff2.b", 0, kOutSlice * r + o);
      for (int o = 0; o < 128; ++o) {
        vl[VL_LN1G + o] = atf(pre + ".ln1.g", 0, o);
        vl[VL_LN1B + o] = atf(pre + ".ln1.b", 0, o);
        vl[VL_LN2G + o] = atf(pre + ".ln2.g", 0, o);
        vl[VL_LN2B + o] = atf(pre + ".ln2.b", 0, o);
      }
    }
    for (int o = 0; o < 64; ++o) {
      v[V_ENT1W + o] = atf("lbs.ent1.w", o, 0);
      v[V_ENT1B + o] = atf("lbs.ent1.b", 0, o);
      v[V_ENT2B + o] = atf("lbs.ent2.b", 0, o);
      v[V_ENTLNG + o] = atf("lbs.ent_ln.g", 0, o);
      v[V_ENTLNB + o] = atf("lbs.ent_ln.b", 0, o);
      v[V_TOKB + o] = atf("lbs.tok.b", 0, o);
    }
    for (int o = 0; o < 128; ++o) v[V_HEADW + o] = atf("lbs.head.w", 0, o);
    v[V_HEADB] = atf("lbs.head.b", 0, 0);
    for (int o = 0; o < kCombSlice; ++o) v[V_COMBB + o] = atf("lbs.comb.b", 0, kCombSlice * r + o);
    // LPS vectors (every rank holds them; rank 0 uses them)
    float* vp = v + V_LPS;
    for (int k = 0; k < 5; ++k)
      for (int o = 0; o < 32; ++o) vp[VP_INT + k * 32 + o] = atf("lps.in.w", o, k);
    for (int o = 0; o < 32; ++o) {
      vp[VP_INB + o] = atf("lps.in.b", 0, o);
      vp[VP_INLNG + o] = atf("lps.in_ln.g", 0, o);
      vp[VP_INLNB + o] = atf("lps.in_ln.b", 0, o);
      vp[VP_HEADW + o] = atf("lps.head.w", 0, o);
    }
    vp[VP_HEADB] = atf("lps.head.b", 0, 0);
    for (int l = 0; l < 2; ++l) {
      const std::string pre = "lps.l" + std::to_string(l);
      float* vl = vp + VP_LAYER0 + l * VP_LAYER_STRIDE;
      for (int o = 0; o < 32; ++o) {
        vl[VPL_LN1G + o] = atf(pre + ".ln1.g", 0, o);
        vl[VPL_LN1B + o] = atf(pre + ".ln1.b", 0, o);
        vl[VPL_OUTB + o] = atf(pre + ".out.b", 0, o);
        vl[VPL_LN2G + o] = atf(pre + ".ln2.g", 0, o);
        vl[VPL_LN2B + o] = atf(pre + ".ln2.b", 0, o);
        vl[VPL_FF2B + o] = atf(pre + ".ff2.b", 0, o);
      }
      for (int o = 0; o < 96; ++o) vl[VPL_QKVB + o] = atf(pre + ".qkv.b", 0, o);
      for (int o = 0; o < 64; ++o) vl[VPL_FF1B + o] = atf(pre + ".ff1.b", 0, o);
    }
  }
  for (int l = 0; l < 2; ++l) {
    const std::string pre = "lps.l" + std::to_string(l);
    uint16_t* wl = lps.data() + l * PL_STRIDE;
    for (int k = 0; k < 32; ++k) {
      for (int o = 0; o < 96; ++o) wl[PL_QKV + k * PL_LDQKV + o] = at(pre + ".qkv.w", o, k);
      for (int o = 0; o < 32; ++o) wl[PL_OUT + k * PL_LDOUT + o] = at(pre + ".out.w", o, k);
      for (int o = 0; o < 64; ++o) wl[PL_FF1 + k * PL_LDFF1 + o] = at(pre + ".ff1.w", o, k);
    }
    for (int k = 0; k < 64; ++k)
      for (int o = 0; o < 32; ++o) wl[PL_FF2 + k * PL_LDFF2 + o] = at(pre + ".ff2.w", o, k);
  }
  // the one-CTA kernel's image (rcta): 128 x 64 swizzled A tiles of W [out][in]
  std::vector<uint16_t> cw(static_cast<size_t>(rcta::kChunks) * rcta::kChunkElems, 0);
  std::vector<float> cv(rcta::S_ELEMS, 0.f);
  {
    using namespace rcta;
    auto chunk = [&](int c) { return cw.data() + static_cast<size_t>(c) * kChunkElems; };
    // chunks c0 + t * nkb + kb: rows [128 t, 128 t + 128) (< outs), inputs [64 kb, 64 kb + 64)
    auto tiles = [&](int c0, const std::string& n, int outs, int ins) {
      const int nt = (outs + 127) / 128, nkb = ins / 64;
      for (int t = 0; t < nt; ++t)
        for (int kb = 0; kb < nkb; ++kb)
          for (int m = 0; m < 128 && 128 * t + m < outs; ++m)
            for (int k = 0; k < 64; ++k)
              chunk(c0 + t * nkb + kb)[tile_off(m, k)] = at(n, 128 * t + m, 64 * kb + k);
    };
    tiles(C_ENT, "lbs.ent2.w", 64, 64);
    tiles(C_COMB, "lbs.comb.w", 128, 128);
    for (int l = 0; l < 2; ++l) {
      const std::string pre = "lbs.l" + std::to_string(l);
      const int base = C_LAYER0 + l * CL_CHUNKS;
      tiles(base + CL_QKV, pre + ".qkv.w", 384, 128);
      tiles(base + CL_OUT, pre + ".out.w", 128, 128);
      tiles(base + CL_FF1, pre + ".ff1.w", 256, 128);
      tiles(base + CL_FF2, pre + ".ff2.w", 128, 256);
      float* vl = cv.data() + S_LAYER0 + l * S_LAYER_STRIDE;
      for (int o = 0; o < 384; ++o) vl[SL_QKVB + o] = atf(pre + ".qkv.b", 0, o);
      for (int o = 0; o < 256; ++o) vl[SL_FF1B + o] = atf(pre + ".ff1.b", 0, o);
      for (int o = 0; o < 128; ++o) {
        vl[SL_OUTB + o] = atf(pre + ".out.b", 0, o);
        vl[SL_FF2B + o] = atf(pre + ".ff2.b", 0, o);
        vl[SL_LN1G + o] = atf(pre + ".ln1.g", 0, o);
        vl[SL_LN1B + o] = atf(pre + ".ln1.b", 0, o);
        vl[SL_LN2G + o] = atf(pre + ".ln2.g", 0, o);
        vl[SL_LN2B + o] = atf(pre + ".ln2.b", 0, o);
      }
    }
    uint16_t* pos = reinterpret_cast<uint16_t*>(cv.data() + S_POS);
    for (int j = 0; j < rcta::kPosRows; ++j)
      for (int o = 0; o < 128; ++o) pos[j * 128 + o] = j < gen_len ? at("lbs.pos", j, o) : 0;
    std::copy(lps.begin(), lps.end(), chunk(C_LPS));
    for (int o = 0; o < 64; ++o) {
      cv[S_ENT1W + o] = atf("lbs.ent1.w", o, 0);
      cv[S_ENT1B + o] = atf("lbs.ent1.b", 0, o);
      cv[S_ENT2B + o] = atf("lbs.ent2.b", 0, o);
      cv[S_ENTLNG + o] = atf("lbs.ent_ln.g", 0, o);
      cv[S_ENTLNB + o] = atf("lbs.ent_ln.b", 0, o);
      cv[S_TOKB + o] = atf("lbs.tok.b", 0, o);
    }
    for (int o = 0; o < 128; ++o) {
      cv[S_COMBB + o] = atf("lbs.comb.b", 0, o);
      cv[S_HEADW + o] = atf("lbs.head.w", 0, o);
    }
    cv[S_HEADB] = atf("lbs.head.b", 0, 0);
    // the LPS vectors: the same as every rank's copy above
    std::copy(vec.begin() + V_LPS, vec.begin() + V_ELEMS, cv.begin() + S_LPS);
  }
  const size_t b_lbs = lbs.size() * 2, b_lps = lps.size() * 2, b_vec = vec.size() * 4;
  const size_t o_lps = (b_lbs + 255) / 256 * 256;
  const size_t o_vec = o_lps + (b_lps + 255) / 256 * 256;
  const size_t o_cw = o_vec + (b_vec + 255) / 256 * 256;
  const size_t o_cv = o_cw + (cw.size() * 2 + 255) / 256 * 256;
  const size_t total = o_cv + cv.size() * 4;
  if (h->d_image) cudaFree(h->d_image);
  h->d_image = nullptr;
  cudaError_t e = cudaMalloc(&h->d_image, total);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaMalloc(router image)");
  if ((e = cudaMemcpy(h->d_image, lbs.data(), b_lbs, cudaMemcpyHostToDevice)) != cudaSuccess ||
      (e = cudaMemcpy(h->d_image + o_lps, lps.data(), b_lps, cudaMemcpyHostToDevice)) != cudaSuccess ||
      (e = cudaMemcpy(h->d_image + o_vec, vec.data(), b_vec, cudaMemcpyHostToDevice)) != cudaSuccess ||
      (e = cudaMemcpy(h->d_image + o_cw, cw.data(), cw.size() * 2, cudaMemcpyHostToDevice)) != cudaSuccess ||
      (e = cudaMemcpy(h->d_image + o_cv, cv.data(), cv.size() * 4, cudaMemcpyHostToDevice)) != cudaSuccess)
    return cuda_fail(h, e, "cudaMemcpy(router image)");
  e = cudaMemcpy(h->d_blob, h->h_blob.data(), h->h_blob.size() * 2, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemcpy(router blob)");
  h->img.lbs_w = reinterpret_cast<const __nv_bfloat16*>(h->d_image);
  h->img.lps_w = reinterpret_cast<const __nv_bfloat16*>(h->d_image + o_lps);
  h->img.vec = reinterpret_cast<const float*>(h->d_image + o_vec);
  h->img.tok_table = h->d_tok;
  h->img.cta_w = reinterpret_cast<const __nv_bfloat16*>(h->d_image + o_cw);
  h->img.cta_vec = reinterpret_cast<const float*>(h->d_image + o_cv);
  return upload_seq_weights(h);
}

ebd_status fold(ebd_handle* h, cudaStream_t st) {
  if (h->w_emb == nullptr) return EBD_OK;
  size_t tok_off = 0;
  for (const auto& t : h->layout) {
    if (t.name == "lbs.tok.w") break;
    tok_off += static_cast<size_t>(t.rows) * t.cols;
  }
  cudaError_t e = launch_fold_tok(reinterpret_cast<const __nv_bfloat16*>(h->d_blob + tok_off),
                                  reinterpret_cast<const __nv_bfloat16*>(h->w_emb), h->d_tok,
                                  h->cfg.vocab, h->cfg.d_base, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "fold kernel");
  return EBD_OK;
}

ebd_status check_args(ebd_handle* h, const ebd_step_args* a, bool need_attn, bool need_lm,
                      bool need_state) {
  if (a == nullptr) return fail(h, EBD_ERR_INVALID_ARG, "args is NULL");
  const ebd_config& c = h->cfg;
  if (a->batch < 0 || a->batch > c.max_batch) return fail(h, EBD_ERR_INVALID_ARG, "batch out of range");
  if (a->rows < 0 || a->rows > c.max_rows) return fail(h, EBD_ERR_INVALID_ARG, "rows out of range");
  if (a->rows > a->batch * c.max_window)
    return fail(h, EBD_ERR_INVALID_ARG, "rows exceed batch * max_window");
  if (need_state) {
    if (!a->cu_rows || !a->row_pos || !a->tokens || !a->mask || !a->in_block || !a->blk_meta)
      return fail(h, EBD_ERR_INVALID_ARG, "cu_rows/row_pos/tokens/mask/in_block/blk_meta must be set");
  }
  if (need_lm) {
    if (!a->hidden || !a->w_lm) return fail(h, EBD_ERR_INVALID_ARG, "hidden and w_lm must be set");
    if (a->w_lm_layout != 0 && a->w_lm_layout != 1)
      return fail(h, EBD_ERR_INVALID_ARG, "w_lm_layout must be 0 or 1");
    if (!aligned(a->hidden, 16) || !aligned(a->w_lm, 16))
      return fail(h, EBD_ERR_INVALID_ARG, "hidden and w_lm must be 16-byte aligned");
  }
  if (need_attn) {
    if (!a->cu_rows || !a->prefix_len || !a->q || !a->k_win || !a->v_win || !a->attn_out ||
        (c.max_prefix > 0 && (!a->k_cache || !a->v_cache)))
      return fail(h, EBD_ERR_INVALID_ARG, "attention needs cu_rows, prefix_len, q, k/v and attn_out");
    if (!aligned(a->k_win, 16) || !aligned(a->v_win, 16) || !aligned(a->q, 16) ||
        !aligned(a->attn_out, 16) ||
        (c.max_prefix > 0 && (!aligned(a->k_cache, 16) || !aligned(a->v_cache, 16))))
      return fail(h, EBD_ERR_INVALID_ARG, "q/k/v/attn_out must be 16-byte aligned");
  }
  if (a->suffix != nullptr && c.max_prefix <= 0)
    return fail(h, EBD_ERR_INVALID_ARG, "a suffix range needs a K/V cache (max_prefix > 0)");
  if (a->kv_append != 0 && a->kv_append != 1)
    return fail(h, EBD_ERR_INVALID_ARG, "kv_append must be 0 or 1");
  if (a->kv_append) {
    if (c.max_prefix <= 0 || !a->k_cache || !a->v_cache || !a->k_win || !a->v_win ||
        !a->row_pos || !a->cu_rows || !a->mask)
      return fail(h, EBD_ERR_INVALID_ARG, "kv_append needs the K/V cache, k_win/v_win, row_pos and mask");
    if (!aligned(a->k_cache, 16) || !aligned(a->v_cache, 16) || !aligned(a->k_win, 16) ||
        !aligned(a->v_win, 16))
      return fail(h, EBD_ERR_INVALID_ARG, "K/V cache and window K/V must be 16-byte aligned");
  }
  return EBD_OK;
}

ebd_status run_attention(ebd_handle* h, const ebd_step_args* a, cudaStream_t st,
                         bool pdl = false, bool wait_prior = false, const unsigned* ready = nullptr,
                         unsigned ready_ticket = 0) {
  const ebd_config& c = h->cfg;
  const int D = c.head_dim, Hkv = c.n_heads_kv;
  CUtensorMap kc, vc, kw, vw;
  const uint64_t R = static_cast<uint64_t>(a->rows);
  const uint64_t Pm = static_cast<uint64_t>(c.max_prefix > 0 ? c.max_prefix : 1);
  const void* kcp = c.max_prefix > 0 ? a->k_cache : a->k_win;  // any valid pointer if no cache
  const void* vcp = c.max_prefix > 0 ? a->v_cache : a->v_win;
  {
    const uint64_t dims[4] = {static_cast<uint64_t>(D), static_cast<uint64_t>(Hkv), Pm,
                              static_cast<uint64_t>(c.max_prefix > 0 ? a->batch : 1)};
    const uint64_t str[3] = {static_cast<uint64_t>(D) * 2, static_cast<uint64_t>(Hkv) * D * 2,
                             Pm * Hkv * D * 2};
    const uint32_t box[4] = {64, 1, 64, 1};
    if (!encode_bf16(&kc, kcp, 4, dims, str, box) || !encode_bf16(&vc, vcp, 4, dims, str, box))
      return fail(h, EBD_ERR_CUDA, "cuTensorMapEncodeTiled (K/V cache) failed");
  }
  {
    const uint64_t dims[3] = {static_cast<uint64_t>(D), static_cast<uint64_t>(Hkv), R};
    const uint64_t str[2] = {static_cast<uint64_t>(D) * 2, static_cast<uint64_t>(Hkv) * D * 2};
    const uint32_t box[3] = {64, 1, 64};
    if (!encode_bf16(&kw, a->k_win, 3, dims, str, box) || !encode_bf16(&vw, a->v_win, 3, dims, str, box))
      return fail(h, EBD_ERR_CUDA, "cuTensorMapEncodeTiled (window K/V) failed");
  }
  AttnParams p{};
  p.B = a->batch;
  p.R = a->rows;
  p.Hq = c.n_heads_q;
  p.Hkv = Hkv;
  p.D = D;
  p.group = c.n_heads_q / Hkv;
  p.max_prefix = c.max_prefix;
  p.max_qtiles = h->attn_max_qtiles;
  p.splits = h->attn_splits;
  p.tc = h->attn_tc;
  p.cu_rows = a->cu_rows;
  p.prefix_len = a->prefix_len;
  p.suffix = c.max_prefix > 0 ? a->suffix : nullptr;
  p.q = reinterpret_cast<const __nv_bfloat16*>(a->q);
  p.out = a->attn_out;
  p.part = h->attn_part;
  p.part_ml = h->attn_part_ml;
  p.tickets = h->tickets;
  p.status = h->d_status;
  p.limit_ns = kLimitNs;
  p.wait_prior = wait_prior ? 1 : 0;
  p.ready = ready;
  p.ready_ticket = ready_ticket;
  if (ready != nullptr && (c.debug_flags & EBD_DEBUG_FORCE_COPY_TIMEOUT)) {
    p.ready_ticket = ready_ticket ^ 0x80000000u;  // never written
    p.limit_ns = 20ull * 1000 * 1000;
  }
  cudaError_t e = launch_attention(kc, vc, kw, vw, p, st, pdl);
  if (e != cudaSuccess) return cuda_fail(h, e, "attention launch");
  return EBD_OK;
}

// pdl_first: the first LM-head launch is a programmatic dependent of the
// kernel just before it on `st`, which copies the hidden rows in.
// v_off, v_count: a->w_lm holds the vocabulary rows [v_off, v_off + v_count)
// (a shard of the vocabulary-parallel LM head); v_count < 0: all of them.
ebd_status run_lm(ebd_handle* h, const ebd_step_args* a, cudaStream_t st, bool pdl_first = false,
                  int v_off = 0, int v_count = -1) {
  const ebd_config& c = h->cfg;
  const int V = v_count < 0 ? c.vocab : v_count;
  CUtensorMap tw;
  const bool packed = a->w_lm_layout == 1;
  if (!encode_w_lm(&tw, a->w_lm, V, c.d_model, packed, 0))
    return fail(h, EBD_ERR_CUDA, "cuTensorMapEncodeTiled (W_lm) failed");
  for (int g0 = 0; g0 < a->rows; g0 += kMaxGroupRows) {
    const int rows = a->rows - g0 < kMaxGroupRows ? a->rows - g0 : kMaxGroupRows;
    LmParams p{};
    // from kLmPairMinRows rows on, CTA pairs run cta_group::2 MMAs of
    // M = 256: each SM receives half of the hidden rows per MMA
    int pair_min = kLmPairMinRows;
    if (const char* env = getenv("EBD_LM_PAIR_MIN")) pair_min = atoi(env) > 0 ? atoi(env) : kMaxGroupRows + 1;
    const int units = (V + kUnit - 1) / kUnit;
    const bool pair = rows >= pair_min && h->grid_lm >= lm_pair_grid(h->num_sms, units);
    lm_plan(p, rows, V, c.d_model, h->num_sms, pair);
    // a shard's own grid may exceed the partial columns of the handle
    if (p.grp_cols > h->grid_lm) lm_plan(p, rows, V, c.d_model, h->grid_lm, pair);
    if (p.grp_cols > h->grid_lm) return fail(h, EBD_ERR_UNSUPPORTED, "LM head: grid exceeds the partials");
    p.ncols = h->grid_lm;
    p.part_rows = c.max_rows;
    p.v_off = v_off;
    if (p.stages < 2) return fail(h, EBD_ERR_UNSUPPORTED, "LM head: shared memory plan failed");
    p.row0 = g0;
    p.packed = packed ? 1 : 0;
    p.part_f = h->part_f;
    p.part_i = h->part_i;
    p.status = h->d_status;
    p.limit_ns = kLimitNs;
    p.force_timeout = (c.debug_flags & EBD_DEBUG_FORCE_TIMEOUT) ? 1 : 0;
    p.pdl = (g0 == 0 && pdl_first) ? 1 : 0;
    CUtensorMap th;
    const uint64_t dims[2] = {static_cast<uint64_t>(c.d_model), static_cast<uint64_t>(a->rows)};
    const uint64_t str[1] = {static_cast<uint64_t>(c.d_model) * 2};
    // a CTA of a pair loads half of each N sub-tile of hidden rows
    const uint32_t box[2] = {64, static_cast<uint32_t>(p.pair ? p.nb / 2 : p.nb)};
    if (!encode_bf16(&th, a->hidden, 2, dims, str, box))
      return fail(h, EBD_ERR_CUDA, "cuTensorMapEncodeTiled (hidden) failed");
    CUtensorMap tw4;  // the paired launches' view of packed W: one box per stage
    if (p.pair && packed && !encode_w_lm(&tw4, a->w_lm, V, c.d_model, packed, p.kbs))
      return fail(h, EBD_ERR_CUDA, "cuTensorMapEncodeTiled (W_lm) failed");
    cudaError_t e = launch_lm_stats(p.pair && packed ? tw4 : tw, th, p, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "LM-head launch");
    h->lm_ctas = p.grid;
  }
  return EBD_OK;
}

// Which kernel decides a launch of `batch` sequences with windows of up to
// kCtaWindow rows: the one-CTA kernel from kCtaMinBatch sequences on, the
// cluster kernel below.  Measured on the LLaDA-8B head shape (µs per step,
// one-CTA against cluster): 1 x 32 rows 209 / 197, 4 x 32 245 / 214,
// 16 x 8 200 / 212, 16 x 32 454 / 465, 64 x 8 464 / 515, 64 x 32 1638 /
// 1749: one sequence decides faster on eight SMs, while many sequences
// need several waves of 8-CTA clusters.  EBD_DECIDE_KERNEL=cta or cluster
// overrides the rule (a measurement knob).
constexpr int kCtaMinBatch = 16;
bool cta_decision(const ebd_handle* h, int batch) {
  if (h->cfg.max_window > kCtaWindow) return false;
  if (const char* env = getenv("EBD_DECIDE_KERNEL")) {
    if (strcmp(env, "cta") == 0) return true;
    if (strcmp(env, "cluster") == 0) return false;
  }
  return batch >= kCtaMinBatch;
}

DecideParams decide_params(ebd_handle* h, const ebd_step_args* a, int features_in) {
  const ebd_config& c = h->cfg;
  DecideParams p{};
  p.B = a->batch;
  p.V = c.vocab;
  p.grid_lm = h->grid_lm;
  p.features_in = features_in;
  p.gen_len = c.gen_len;
  p.g_max = c.g_max;
  p.l_min = c.l_min;
  p.l_b = c.l_b;
  p.eos_id = c.eos_id;
  p.mode = c.decode_mode;
  p.top_m = c.top_m;
  p.lps_enabled = c.decode_mode == EBD_DECODE_EB ? c.lps_enabled : 0;
  p.tau = c.tau;
  p.tau_psi = c.tau_psi;
  p.inv_log_v = static_cast<float>(1.0 / std::log(static_cast<double>(c.vocab)));
  p.cu_rows = a->cu_rows;
  p.row_pos = a->row_pos;
  p.part_f = h->part_f;
  p.part_i = h->part_i;
  p.tokens = a->tokens;
  p.mask = a->mask;
  p.in_block = a->in_block;
  p.blk_meta = a->blk_meta;
  p.tokens_out = a->tokens;
  p.mask_out = a->mask;
  p.in_block_out = a->in_block;
  p.blk_meta_out = a->blk_meta;
  p.conf = a->conf;
  p.entropy = a->entropy;
  p.ent_norm = a->ent_norm;
  p.gap = a->gap;
  p.argmax = a->argmax;
  p.lbs_logit = a->lbs_logit;
  p.lps_prob = a->lps_prob;
  p.accepted = a->accepted;
  p.status = h->d_status;
  p.rows_expected = a->rows;
  p.w = h->img;
  return p;
}

}  // namespace

extern "C" {

const char* ebd_version(void) { return "ebd 0.1 (sm_103a)"; }

ebd_status ebd_loop_block_window(const uint8_t* mask, int32_t L, int32_t block, int32_t* lo,
                                 int32_t* hi) {
  if (mask == nullptr || lo == nullptr || hi == nullptr || L < 0 || block < 1)
    return EBD_ERR_INVALID_ARG;
  for (int32_t j0 = 0; j0 < L; j0 += block) {
    const int32_t j1 = j0 + block < L ? j0 + block : L;
    for (int32_t i = j0; i < j1; ++i)
      if (mask[i]) {
        *lo = j0;
        *hi = j1;
        return EBD_OK;
      }
  }
  *lo = *hi = L;
  return EBD_OK;
}

ebd_status ebd_loop_window(const uint8_t* mask, const uint8_t* in_block, const int32_t* meta,
                           int32_t L, int32_t max_window, int32_t* lo, int32_t* hi) {
  if (mask == nullptr || in_block == nullptr || meta == nullptr || lo == nullptr || hi == nullptr ||
      L < 0 || max_window < 1)
    return EBD_ERR_INVALID_ARG;
  int32_t f = L;
  for (int32_t i = 0; i < L; ++i)
    if (mask[i]) {
      f = i;
      break;
    }
  if (f == L) {
    *lo = *hi = L;
    return EBD_OK;
  }
  int32_t end;
  if (meta[1] == 0) {
    end = f + max_window < L ? f + max_window : L;
  } else {
    int32_t last = -1;
    for (int32_t i = L - 1; i >= 0; --i)
      if (in_block[i]) {
        last = i;
        break;
      }
    if (last < 0) return EBD_ERR_STATE;
    end = last + 1;
    if (end <= f || end - f > max_window) return EBD_ERR_STATE;
  }
  *lo = f;
  *hi = end;
  return EBD_OK;
}

size_t ebd_weight_count(const ebd_config* cfg) {
  if (cfg == nullptr || cfg->d_base <= 0 || cfg->gen_len <= 0) return 0;
  return layout_count(router_layout(cfg->d_base, cfg->gen_len));
}

ebd_status ebd_router_init_host(const ebd_config* cfg, void* host, size_t* bytes) {
  if (cfg == nullptr || bytes == nullptr) return EBD_ERR_INVALID_ARG;
  if (cfg->d_base <= 0 || cfg->gen_len <= 0) return EBD_ERR_UNSUPPORTED;
  const auto layout = router_layout(cfg->d_base, cfg->gen_len);
  const size_t need = layout_count(layout) * 2;
  if (host == nullptr) {
    *bytes = need;
    return EBD_OK;
  }
  if (*bytes < need) return EBD_ERR_INVALID_ARG;
  router_init(cfg->seed, layout, static_cast<uint16_t*>(host));
  *bytes = need;
  return EBD_OK;
}

ebd_status ebd_create(const ebd_config* cfg, ebd_handle** out) {
  if (out == nullptr) return EBD_ERR_INVALID_ARG;
  *out = nullptr;
  if (cfg == nullptr) return EBD_ERR_INVALID_ARG;
  std::string why;
  ebd_status s = validate_config(cfg, why);
  if (s != EBD_OK) {
    std::fprintf(stderr, "ebd_create: %s\n", why.c_str());
    return s;
  }
  ebd_handle* h = new ebd_handle();
  h->cfg = *cfg;
  auto bail = [&](ebd_status code) {
    std::fprintf(stderr, "ebd_create: %s\n", h->err.c_str());
    ebd_destroy(h);
    return code;
  };
  cudaError_t e = cudaGetDevice(&h->device);
  if (e != cudaSuccess) return bail(cuda_fail(h, e, "cudaGetDevice"));
  e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
  if (e != cudaSuccess) return bail(cuda_fail(h, e, "cudaDeviceGetAttribute"));
  int cc_major = 0, cc_minor = 0;
  cudaDeviceGetAttribute(&cc_major, cudaDevAttrComputeCapabilityMajor, h->device);
  cudaDeviceGetAttribute(&cc_minor, cudaDevAttrComputeCapabilityMinor, h->device);
  if (cc_major != 10 || cc_minor != 3)
    return bail(fail(h, EBD_ERR_UNSUPPORTED, "the library is compiled for sm_103a (GB300) only"));
  if (get_encode() == nullptr)
    return bail(fail(h, EBD_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable"));
  if ((e = lm_configure()) != cudaSuccess) return bail(cuda_fail(h, e, "LM-head attributes"));
  if ((e = attn_configure()) != cudaSuccess) return bail(cuda_fail(h, e, "attention attributes"));
  if ((e = decide_configure()) != cudaSuccess || (e = decide_cta_configure()) != cudaSuccess)
    return bail(cuda_fail(h, e, "decision attributes"));

  h->layout = router_layout(cfg->d_base, cfg->gen_len);
  h->h_blob.resize(layout_count(h->layout));
  router_init(cfg->seed, h->layout, h->h_blob.data());
  if ((e = cudaMalloc(&h->d_blob, h->h_blob.size() * 2)) != cudaSuccess)
    return bail(cuda_fail(h, e, "cudaMalloc(router blob)"));
  if ((e = cudaMalloc(&h->d_tok, static_cast<size_t>(cfg->vocab) * 64 * 4)) != cudaSuccess)
    return bail(cuda_fail(h, e, "cudaMalloc(token table)"));
  if ((s = upload_router(h)) != EBD_OK) return bail(s);

  // LM-head partials: one state per (row, CTA)
  h->lm_units = (cfg->vocab + kUnit - 1) / kUnit;
  h->grid_lm = lm_grid(h->num_sms, h->lm_units);
  {  // a handle whose steps may take the paired LM head leaves room for its partials
    int pair_min = kLmPairMinRows;
    if (const char* env = getenv("EBD_LM_PAIR_MIN")) pair_min = atoi(env) > 0 ? atoi(env) : kMaxGroupRows + 1;
    const int pg = lm_pair_grid(h->num_sms, h->lm_units);
    if (cfg->max_rows >= pair_min && pg > h->grid_lm) h->grid_lm = pg;
  }
  const size_t np = static_cast<size_t>(cfg->max_rows) * h->grid_lm;
  if ((e = cudaMalloc(&h->part_f, np * sizeof(float4))) != cudaSuccess)
    return bail(cuda_fail(h, e, "cudaMalloc(partials)"));
  if ((e = cudaMalloc(&h->part_i, np * sizeof(int))) != cudaSuccess)
    return bail(cuda_fail(h, e, "cudaMalloc(partials)"));
  // attention split-KV workspace
  {
    // Both attention kernels take 64-row query tiles.  The tcgen05 kernel
    // holds an SM alone (one CTA per SM) and pays a fixed setup and drain
    // per CTA (TMEM, barriers, the query tile, its output), which long key
    // ranges amortise; the mma.sync kernel runs two CTAs per SM and keeps
    // launches of many short key ranges (measured, attention alone, LLaDA-8B
    // heads, us, mma.sync against tcgen05: 16 x 256 x 32 rows 41.6 / 47.8,
    // 64 x 1024 x 8 211.6 / 230.0; but 16 x 4096 x 32 305.8 / 203.4,
    // 64 x 4096 x 32 1032.9 / 690.8, 4 x 1024 x 32 45.7 / 27.3, LLaDA-8B
    // 21.2 / 17.1, Dream-7B 53.9 / 39.6).  EBD_ATTN_KERNEL=tc|mma forces one,
    // EBD_ATTN_SPLITS the split count (measurement sweeps).
    const int tile = 64;
    const int group = cfg->n_heads_q / cfg->n_heads_kv;
    const int aw = cfg->max_window < kMaxWindow ? cfg->max_window : kMaxWindow;
    h->attn_max_qtiles = (aw * group + tile - 1) / tile;
    const int slots = cfg->max_batch * cfg->n_heads_kv * h->attn_max_qtiles;
    const int nch = (cfg->max_prefix + kAttnChunk - 1) / kAttnChunk + 1;
    h->attn_tc = (slots <= 2 * h->num_sms || nch >= 65 || (nch >= 17 && aw >= 32)) ? 1 : 0;
    if (const char* env = getenv("EBD_ATTN_KERNEL")) h->attn_tc = strcmp(env, "mma") == 0 ? 0 : 1;
    int splits;
    if (h->attn_tc) {
      // one split, unless few tiles leave most SMs idle: then about one
      // CTA per SM, but at least 8 key chunks per split
      splits = 1;
      if (2 * slots < h->num_sms) {
        splits = (h->num_sms + slots - 1) / slots;
        if (splits > nch / 8) splits = nch / 8;
      }
    } else {
      splits = (2 * h->num_sms + slots - 1) / slots;
    }
    if (const char* env = getenv("EBD_ATTN_SPLITS")) splits = atoi(env);
    if (splits > kMaxSplits) splits = kMaxSplits;
    if (splits > nch) splits = nch;
    if (splits < 1) splits = 1;
    h->attn_splits = splits;
    if (splits > 1) {
      const size_t bytes = static_cast<size_t>(slots) * splits * tile * (cfg->head_dim + 2) * 4;
      if ((e = cudaMalloc(&h->attn_part, bytes)) != cudaSuccess)
        return bail(cuda_fail(h, e, "cudaMalloc(attention partials)"));
      h->attn_part_ml = h->attn_part + static_cast<size_t>(slots) * splits * tile * cfg->head_dim;
    }
    if ((e = cudaMalloc(&h->tickets, static_cast<size_t>(slots) * sizeof(int))) != cudaSuccess)
      return bail(cuda_fail(h, e, "cudaMalloc(tickets)"));
    if ((e = cudaMemset(h->tickets, 0, static_cast<size_t>(slots) * sizeof(int))) != cudaSuccess)
      return bail(cuda_fail(h, e, "cudaMemset(tickets)"));
  }
  if ((e = cudaMalloc(&h->d_status, sizeof(int))) != cudaSuccess)
    return bail(cuda_fail(h, e, "cudaMalloc(status)"));
  if ((e = cudaMemset(h->d_status, 0, sizeof(int))) != cudaSuccess)
    return bail(cuda_fail(h, e, "cudaMemset(status)"));
  // staging for ebd_step_host
  {
    const size_t R = cfg->max_rows, B = cfg->max_batch;
    const size_t d = cfg->d_model, Hq = cfg->n_heads_q, Hkv = cfg->n_heads_kv, D = cfg->head_dim;
    size_t bytes = 0;
    auto add = [&](size_t n) { bytes += (n + 255) / 256 * 256; };
    add((B + 1) * 4); add(B * 4); add(R * 4); add(R * d * 2); add(R * Hq * D * 2);
    add(R * Hkv * D * 2); add(R * Hkv * D * 2); add(R * 4); add(R); add(R); add(B * 8);
    add(R * Hq * D * 4); for (int i = 0; i < 6; ++i) add(R * 4); add(R * 4); add(R);
    add(B * 8);  // suffix ranges
    h->staging_bytes = bytes;
    if ((e = cudaMalloc(&h->staging, bytes)) != cudaSuccess)
      return bail(cuda_fail(h, e, "cudaMalloc(staging)"));
  }
  // the copy stream of ebd_step_host, set up here rather than at its first
  // call, which may come while a stream is being captured into a graph
  if (cfg->max_window <= kMaxWindow) (void)copy_route_ready(h);
  if (cfg->max_window > kMaxWindow) {  // scratch of the grid-wide decision
    const size_t R = cfg->max_rows, B = cfg->max_batch;
    size_t bytes = 0;
    auto add = [&](size_t n) {
      const size_t at = bytes;
      bytes += (n + 255) / 256 * 256;
      return at;
    };
    const size_t o_conf = add(R * 4), o_entn = add(R * 4), o_gap = add(R * 4), o_arg = add(R * 4);
    const size_t o_seq = add(R * 4), o_mr = add(R * 4), o_mrows = add(R * 4), o_bmr = add(R * 4),
                 o_bmrows = add(R * 4), o_bad = add(R), o_ib = add(R), o_sq = add((B + 1) * 8 * 4),
                 o_O = add(R * 4), o_P = add(R * 4), o_f = add(R * 8 * 4), o_Z = add(R * 128 * 4),
                 o_QKV = add(R * 384 * 4), o_A = add(R * 128 * 4), o_Zp = add(R * 32 * 4),
                 o_QKVp = add(R * 96 * 4), o_Ap = add(R * 32 * 4);
    if ((e = cudaMalloc(&h->seq_scratch, bytes)) != cudaSuccess)
      return bail(cuda_fail(h, e, "cudaMalloc(decision scratch)"));
    uint8_t* b0 = h->seq_scratch;
    SeqParams& q = h->seqp;
    q.conf = reinterpret_cast<float*>(b0 + o_conf);
    q.ent_norm = reinterpret_cast<float*>(b0 + o_entn);
    q.gap = reinterpret_cast<float*>(b0 + o_gap);
    q.argmax = reinterpret_cast<int*>(b0 + o_arg);
    q.seq_of = reinterpret_cast<int*>(b0 + o_seq);
    q.mrank = reinterpret_cast<int*>(b0 + o_mr);
    q.mrows = reinterpret_cast<int*>(b0 + o_mrows);
    q.bmrank = reinterpret_cast<int*>(b0 + o_bmr);
    q.bmrows = reinterpret_cast<int*>(b0 + o_bmrows);
    q.bad = b0 + o_bad;
    q.ib = b0 + o_ib;
    q.sq = reinterpret_cast<int*>(b0 + o_sq);
    q.O = reinterpret_cast<float*>(b0 + o_O);
    q.P = reinterpret_cast<float*>(b0 + o_P);
    q.feats = reinterpret_cast<float*>(b0 + o_f);
    q.Z = reinterpret_cast<float*>(b0 + o_Z);
    q.QKV = reinterpret_cast<float*>(b0 + o_QKV);
    q.A = reinterpret_cast<float*>(b0 + o_A);
    q.Zp = reinterpret_cast<float*>(b0 + o_Zp);
    q.QKVp = reinterpret_cast<float*>(b0 + o_QKVp);
    q.Ap = reinterpret_cast<float*>(b0 + o_Ap);
  }
  for (int i = 0; i < 4; ++i)
    if ((e = cudaEventCreate(&h->ev[i])) != cudaSuccess)
      return bail(cuda_fail(h, e, "cudaEventCreate"));
  if ((e = cudaDeviceSynchronize()) != cudaSuccess) return bail(cuda_fail(h, e, "create"));
  *out = h;
  return EBD_OK;
}

void ebd_destroy(ebd_handle* h) {
  if (h == nullptr) return;
  int prev = -1;
  cudaGetDevice(&prev);
  if (prev != h->device) cudaSetDevice(h->device);
  cudaDeviceSynchronize();
  if (h->s_copy) cudaStreamDestroy(h->s_copy);
  if (h->ev_fork) cudaEventDestroy(h->ev_fork);
  if (h->ev_join) cudaEventDestroy(h->ev_join);
  cudaFree(h->d_ready);
  cudaFree(h->d_blob);
  cudaFree(h->d_image);
  cudaFree(h->d_tok);
  cudaFree(h->part_f);
  cudaFree(h->part_i);
  cudaFree(h->attn_part);
  cudaFree(h->tickets);
  cudaFree(h->d_status);
  cudaFree(h->staging);
  cudaFree(h->d_seqw);
  cudaFree(h->seq_scratch);
  for (int i = 0; i < 4; ++i)
    if (h->ev[i]) cudaEventDestroy(h->ev[i]);
  if (prev >= 0 && prev != h->device) cudaSetDevice(prev);
  delete h;
}

const char* ebd_last_error(const ebd_handle* h) { return h ? h->err.c_str() : "null handle"; }

ebd_status ebd_bind_embedding(ebd_handle* h, const uint16_t* w_emb, void* stream) {
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  if (w_emb == nullptr || !aligned(w_emb, 16))
    return fail(h, EBD_ERR_INVALID_ARG, "w_emb must be a 16-byte aligned device pointer");
  h->w_emb = w_emb;
  return fold(h, static_cast<cudaStream_t>(stream));
}

ebd_status ebd_export_weights(const ebd_handle* h, void* host, size_t* bytes) {
  if (h == nullptr || bytes == nullptr) return EBD_ERR_INVALID_ARG;
  const size_t need = h->h_blob.size() * 2;
  if (host == nullptr) {
    *bytes = need;
    return EBD_OK;
  }
  if (*bytes < need) return EBD_ERR_INVALID_ARG;
  std::memcpy(host, h->h_blob.data(), need);
  *bytes = need;
  return EBD_OK;
}

ebd_status ebd_import_weights(ebd_handle* h, const void* host, size_t bytes) {
  if (h == nullptr || host == nullptr) return EBD_ERR_INVALID_ARG;
  if (bytes != h->h_blob.size() * 2) return fail(h, EBD_ERR_INVALID_ARG, "weight blob size mismatch");
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(h, e, "import");
  std::memcpy(h->h_blob.data(), host, bytes);
  if ((s = upload_router(h)) != EBD_OK) return s;
  if ((s = fold(h, nullptr)) != EBD_OK) return s;
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(h, e, "import");
  return EBD_OK;
}

size_t ebd_lm_head_packed_bytes(const ebd_config* cfg) {
  if (cfg == nullptr || cfg->vocab <= 0 || cfg->d_model <= 0) return 0;
  const size_t units = (static_cast<size_t>(cfg->vocab) + kUnit - 1) / kUnit;
  const size_t nkb = (static_cast<size_t>(cfg->d_model) + 63) / 64;
  return units * nkb * 64 * 64 * 2;
}

ebd_status ebd_pack_lm_head(ebd_handle* h, const uint16_t* w_lm, uint16_t* w_packed,
                            void* stream) {
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  if (w_lm == nullptr || w_packed == nullptr || !aligned(w_lm, 16) || !aligned(w_packed, 16))
    return fail(h, EBD_ERR_INVALID_ARG, "w_lm and w_packed must be 16-byte aligned device pointers");
  (void)cudaGetLastError();
  cudaError_t e = launch_pack_lm(reinterpret_cast<const __nv_bfloat16*>(w_lm),
                                 reinterpret_cast<__nv_bfloat16*>(w_packed), h->cfg.vocab,
                                 h->cfg.d_model, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "pack launch");
  return EBD_OK;
}

namespace {
// ebd_step_host moves its inputs in and its results out with one kernel
// each way where the host buffers are pinned and mapped into the device's
// address space (cudaHostAlloc / cudaHostRegister memory): one launch
// instead of a dozen small copies.  Other host buffers are copied with
// cudaMemcpyAsync.
struct CopyItem {
  const uint8_t* src;
  uint8_t* dst;
  uint32_t bytes;
};
constexpr int kMaxCopyItems = 16;
struct CopyList {
  CopyItem it[kMaxCopyItems];
  int n;
};

// A kernel launched after it as a programmatic dependent (the LM head of
// ebd_step_host) may be scheduled at once; it waits for this grid before it
// reads what this one copies.
__global__ void __launch_bounds__(256) copy_list_kernel(const CopyList cl) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int i = blockIdx.y;
  if (i >= cl.n) return;
  const CopyItem c = cl.it[i];
  const size_t stride = static_cast<size_t>(gridDim.x) * blockDim.x;
  const size_t t0 = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const bool vec = ((reinterpret_cast<uintptr_t>(c.src) | reinterpret_cast<uintptr_t>(c.dst) | c.bytes) & 15u) == 0;
  if (vec) {
    const size_t n = c.bytes / 16;
    for (size_t k = t0; k < n; k += stride)
      reinterpret_cast<uint4*>(c.dst)[k] = reinterpret_cast<const uint4*>(c.src)[k];
  } else {
    for (size_t k = t0; k < c.bytes; k += stride) c.dst[k] = c.src[k];
  }
}

// the device address of a pinned, mapped host buffer, else null
const void* mapped_host(const void* host) {
  if (host == nullptr) return nullptr;
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, host) != cudaSuccess) {
    (void)cudaGetLastError();
    return nullptr;
  }
  return at.type == cudaMemoryTypeHost ? at.devicePointer : nullptr;
}

// copies (dst, src, bytes): mapped host buffers go to one copy_list_kernel,
// the others to cudaMemcpyAsync
struct HostMover {
  cudaStream_t st;
  bool to_device;
  CopyList list{};
  cudaError_t err = cudaSuccess;
  void add(void* dst, const void* src, size_t bytes) {
    if (bytes == 0 || dst == nullptr || src == nullptr || err != cudaSuccess) return;
    const void* host = to_device ? src : dst;
    const void* dev = mapped_host(host);
    if (dev != nullptr && list.n < kMaxCopyItems && bytes < (1ull << 31)) {
      CopyItem& c = list.it[list.n++];
      c.src = static_cast<const uint8_t*>(to_device ? dev : src);
      c.dst = static_cast<uint8_t*>(to_device ? dst : const_cast<void*>(dev));
      c.bytes = static_cast<uint32_t>(bytes);
      return;
    }
    err = cudaMemcpyAsync(dst, src, bytes, to_device ? cudaMemcpyHostToDevice : cudaMemcpyDeviceToHost, st);
  }
  cudaError_t flush() {
    if (err != cudaSuccess || list.n == 0) return err;
    uint32_t most = 0;
    for (int i = 0; i < list.n; ++i) most = list.it[i].bytes > most ? list.it[i].bytes : most;
    unsigned bx = (most + 16 * 256 - 1) / (16 * 256);
    bx = bx < 1 ? 1 : (bx > 64 ? 64 : bx);
    copy_list_kernel<<<dim3(bx, static_cast<unsigned>(list.n)), 256, 0, st>>>(list);
    list.n = 0;
    return cudaGetLastError();
  }
};

// What ebd_step_host changes in a step: the ticket the attention waits for
// (its inputs come in on the copy stream) and where the decision writes the
// decode state (the caller's buffers, when it read a staged copy).
struct StepRoute {
  bool lm_pdl;  // the kernel just before the step copied the hidden rows in
  const unsigned* ready;
  unsigned ready_ticket;
  int* tokens_out;
  uint8_t* mask_out;
  uint8_t* in_block_out;
  int* blk_meta_out;
};

}  // namespace

namespace {
// windows of more than kMaxWindow rows per sequence: the grid-wide decision
bool seq_mode(const ebd_handle* h) { return h->cfg.max_window > kMaxWindow; }

SeqParams seq_params(ebd_handle* h, const ebd_step_args* a, const float* conf,
                     const float* ent_norm, const float* gap, const int* argmax) {
  const ebd_config& c = h->cfg;
  SeqParams p = h->seqp;  // scratch
  p.B = a->batch;
  p.R = a->rows;
  p.V = c.vocab;
  p.gen_len = c.gen_len;
  p.g_max = c.g_max;
  p.l_min = c.l_min;
  p.l_b = c.l_b;
  p.eos_id = c.eos_id;
  p.mode = c.decode_mode;
  p.top_m = c.top_m;
  p.lps_enabled = c.decode_mode == EBD_DECODE_EB ? c.lps_enabled : 0;
  p.tau = c.tau;
  p.tau_psi = c.tau_psi;
  p.cu_rows = a->cu_rows;
  p.row_pos = a->row_pos;
  p.tokens = a->tokens;
  p.mask = a->mask;
  p.in_block = a->in_block;
  p.blk_meta = a->blk_meta;
  p.conf = conf;
  p.ent_norm = ent_norm;
  p.gap = gap;
  p.argmax = argmax;
  p.accepted = a->accepted;
  p.lbs_logit = a->lbs_logit;
  p.lps_prob = a->lps_prob;
  p.w = h->d_seqw;
  p.o = h->seqw;
  p.tok_table = h->d_tok;
  p.status = h->d_status;
  return p;
}

// LM head, merge into the statistics, grid-wide decision
ebd_status step_seq(ebd_handle* h, const ebd_step_args* a, cudaStream_t st) {
  if (a->attn_out != nullptr || a->kv_append)
    return fail(h, EBD_ERR_UNSUPPORTED,
                "the window attention and the cache append need windows of at most 64 rows "
                "(this handle has max_window > 64)");
  const int prof = h->profile;
  cudaError_t e;
  float* conf = a->conf ? a->conf : const_cast<float*>(h->seqp.conf);
  float* entn = a->ent_norm ? a->ent_norm : const_cast<float*>(h->seqp.ent_norm);
  float* gap = a->gap ? a->gap : const_cast<float*>(h->seqp.gap);
  int* arg = a->argmax ? a->argmax : const_cast<int*>(h->seqp.argmax);
  const SeqParams sp = seq_params(h, a, conf, entn, gap, arg);
  // the decision's scratch reset first: from the LM head on, every kernel is
  // a programmatic dependent of the one before it (unless profiled)
  if ((e = launch_decide_seq_init(sp, st)) != cudaSuccess) return cuda_fail(h, e, "decision reset");
  if (prof && (e = record(h->ev[0], st)) != cudaSuccess) return cuda_fail(h, e, "profile event");
  ebd_status s = run_lm(h, a, st);
  if (s != EBD_OK) return s;
  if (prof && (e = record(h->ev[1], st)) != cudaSuccess) return cuda_fail(h, e, "profile event");
  const float inv = static_cast<float>(1.0 / std::log(static_cast<double>(h->cfg.vocab)));
  if ((e = launch_merge_stats(h->part_f, h->part_i, a->rows, h->grid_lm, h->cfg.vocab, inv, conf,
                              a->entropy, entn, gap, arg, h->d_status, st, prof == 0)) != cudaSuccess)
    return cuda_fail(h, e, "merge launch");
  if ((e = launch_decide_seq(sp, st, true)) != cudaSuccess) return cuda_fail(h, e, "decision launch");
  if (prof && (e = record(h->ev[2], st)) != cudaSuccess) return cuda_fail(h, e, "profile event");
  if (prof && (e = record(h->ev[3], st)) != cudaSuccess) return cuda_fail(h, e, "profile event");
  h->prof_mode = prof;
  h->prof_attn = 0;
  return EBD_OK;
}
}  // namespace

namespace {
// One step of the block-window setting (windows of at most kMaxWindow rows).
// Order on `st`: LM head, decision, window attention, (cache append).  The
// attention feeds neither of the others, so unless every kernel is timed on
// its own (profile mode 1) it is launched as a programmatic dependent of the
// decision: it fills the SMs the decision's clusters leave idle.  The append
// reads the mask the decision writes: it is a programmatic dependent of the
// attention and waits for it, and the attention, in that case, waits for the
// decision before it exits.  The attention reads no cache position the
// append writes.
ebd_status step_run(ebd_handle* h, const ebd_step_args* a, cudaStream_t st, const StepRoute* rt) {
  const bool attn = a->attn_out != nullptr;
  ebd_status s;
  const int prof = h->profile;
  cudaError_t e0 = cudaSuccess;
  if (prof && (e0 = record(h->ev[0], st)) != cudaSuccess) return cuda_fail(h, e0, "profile event");
  if ((s = run_lm(h, a, st, rt != nullptr && rt->lm_pdl && prof == 0)) != EBD_OK) return s;
  if (prof && (e0 = record(h->ev[1], st)) != cudaSuccess) return cuda_fail(h, e0, "profile event");
  DecideParams p = decide_params(h, a, 0);
  p.pdl = prof == 0 ? 1 : 0;  // no event between the LM head and the decision
  if (rt != nullptr) {
    p.tokens_out = rt->tokens_out;
    p.mask_out = rt->mask_out;
    p.in_block_out = rt->in_block_out;
    p.blk_meta_out = rt->blk_meta_out;
  }
  const bool cta = cta_decision(h, a->batch);
  // the LM head's CTAs hold one SM each: the decision's CTAs are placed while
  // it runs if enough SMs are left, and then warm up on a stand-in window
  p.warm = (p.pdl && cta && h->num_sms - h->lm_ctas >= a->batch) ? 1 : 0;
  cudaError_t e = cta ? launch_decide_cta(p, st) : launch_decide(p, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "decision launch");
  if (prof == 1 && (e0 = record(h->ev[2], st)) != cudaSuccess)
    return cuda_fail(h, e0, "profile event");
  const bool pdl_attn = prof != 1;
  if (attn && (s = run_attention(h, a, st, pdl_attn, a->kv_append != 0, rt ? rt->ready : nullptr,
                                 rt ? rt->ready_ticket : 0u)) != EBD_OK)
    return s;
  if (a->kv_append) {
    const ebd_config& c = h->cfg;
    // a programmatic dependent only of a kernel that waits for the decision
    e = launch_kv_append(a->k_cache, a->v_cache, a->k_win, a->v_win, a->cu_rows, a->row_pos,
                         rt != nullptr ? rt->mask_out : a->mask, a->batch, a->rows, c.max_prefix,
                         c.n_heads_kv * c.head_dim, st, attn && pdl_attn);
    if (e != cudaSuccess) return cuda_fail(h, e, "cache append launch");
  }
  if (prof && (e0 = record(h->ev[3], st)) != cudaSuccess) return cuda_fail(h, e0, "profile event");
  h->prof_mode = prof;
  h->prof_attn = attn ? 1 : 0;
  return EBD_OK;
}
}  // namespace

ebd_status ebd_step(ebd_handle* h, const ebd_step_args* a, void* stream) {
  NvtxRange nvtx("ebd_step");
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  const bool attn = a != nullptr && a->attn_out != nullptr;
  if ((s = check_args(h, a, attn, true, true)) != EBD_OK) return s;
  if (h->w_emb == nullptr) return fail(h, EBD_ERR_STATE, "bind the token embedding first");
  if (a->rows == 0 || a->batch == 0) return EBD_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  (void)cudaGetLastError();  // a stale error of an earlier unrelated call is not ours
  if (seq_mode(h)) return step_seq(h, a, st);
  return step_run(h, a, st, nullptr);
}

ebd_status ebd_decide(ebd_handle* h, const ebd_step_args* a, void* stream) {
  NvtxRange nvtx("ebd_decide");
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  if ((s = check_args(h, a, false, false, true)) != EBD_OK) return s;
  if (!a->conf || !a->ent_norm || !a->gap || !a->argmax)
    return fail(h, EBD_ERR_INVALID_ARG, "conf/ent_norm/gap/argmax inputs must be set");
  if (h->w_emb == nullptr) return fail(h, EBD_ERR_STATE, "bind the token embedding first");
  if (a->rows == 0 || a->batch == 0) return EBD_OK;
  if (seq_mode(h)) {
    const SeqParams sp = seq_params(h, a, a->conf, a->ent_norm, a->gap, a->argmax);
    cudaError_t e = launch_decide_seq_init(sp, static_cast<cudaStream_t>(stream));
    if (e == cudaSuccess) e = launch_decide_seq(sp, static_cast<cudaStream_t>(stream), false);
    if (e != cudaSuccess) return cuda_fail(h, e, "decision launch");
    return EBD_OK;
  }
  DecideParams p = decide_params(h, a, 1);
  p.entropy = nullptr;
  cudaError_t e = cta_decision(h, a->batch) ? launch_decide_cta(p, static_cast<cudaStream_t>(stream))
                                  : launch_decide(p, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "decision launch");
  return EBD_OK;
}

ebd_status ebd_lm_stats(ebd_handle* h, const ebd_step_args* a, void* stream) {
  NvtxRange nvtx("ebd_lm_stats");
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  if ((s = check_args(h, a, false, true, false)) != EBD_OK) return s;
  if (a->rows == 0) return EBD_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if ((s = run_lm(h, a, st)) != EBD_OK) return s;
  const float inv = static_cast<float>(1.0 / std::log(static_cast<double>(h->cfg.vocab)));
  cudaError_t e = launch_merge_stats(h->part_f, h->part_i, a->rows, h->grid_lm, h->cfg.vocab, inv,
                                     a->conf, a->entropy, a->ent_norm, a->gap, a->argmax,
                                     h->d_status, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "merge launch");
  return EBD_OK;
}

ebd_status ebd_lm_shard_state(ebd_handle* h, const ebd_step_args* a, int32_t v_off,
                              int32_t v_count, float* state, void* stream) {
  NvtxRange nvtx("ebd_lm_shard_state");
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  if ((s = check_args(h, a, false, true, false)) != EBD_OK) return s;
  if (v_off < 0 || v_count < 1 || v_off % kUnit != 0 || v_count > h->cfg.vocab - v_off)
    return fail(h, EBD_ERR_INVALID_ARG, "shard range: v_off a multiple of 64, within the vocabulary");
  if (a->rows == 0) return EBD_OK;
  if (state == nullptr || !aligned(state, 16))
    return fail(h, EBD_ERR_INVALID_ARG, "state must be a 16-byte aligned device pointer");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if ((s = run_lm(h, a, st, false, v_off, v_count)) != EBD_OK) return s;
  cudaError_t e = launch_shard_state(h->part_f, h->part_i, a->rows, h->grid_lm, state, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "shard state launch");
  return EBD_OK;
}

ebd_status ebd_merge_shard_states(ebd_handle* h, const float* states, int32_t shards,
                                  const ebd_step_args* a, void* stream) {
  NvtxRange nvtx("ebd_merge_shard_states");
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  if (a == nullptr) return fail(h, EBD_ERR_INVALID_ARG, "args is NULL");
  if (a->rows < 0 || a->rows > h->cfg.max_rows) return fail(h, EBD_ERR_INVALID_ARG, "rows out of range");
  if (shards < 1) return fail(h, EBD_ERR_INVALID_ARG, "shards must be >= 1");
  if (a->rows == 0) return EBD_OK;
  if (states == nullptr || !aligned(states, 16))
    return fail(h, EBD_ERR_INVALID_ARG, "states must be a 16-byte aligned device pointer");
  const float inv = static_cast<float>(1.0 / std::log(static_cast<double>(h->cfg.vocab)));
  cudaError_t e = launch_merge_shards(states, shards, a->rows, h->cfg.vocab, inv, a->conf, a->entropy,
                                      a->ent_norm, a->gap, a->argmax, h->d_status,
                                      static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "shard merge launch");
  return EBD_OK;
}

ebd_status ebd_attention(ebd_handle* h, const ebd_step_args* a, void* stream) {
  NvtxRange nvtx("ebd_attention");
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  if ((s = check_args(h, a, true, false, false)) != EBD_OK) return s;
  if (a->rows == 0 || a->batch == 0) return EBD_OK;
  return run_attention(h, a, static_cast<cudaStream_t>(stream));
}


// In the block-window setting the results go straight into the caller's
// mapped host buffers (the kernels' stores cross the host link; nothing is
// copied back after the step), and with the attention, its own inputs (q and
// the window K/V, which nothing else before it reads) come in on a copy
// engine while the LM head runs: a second stream, forked after the copy of
// what the LM head and the decision read, copies them and then writes the
// step's ticket, which the attention waits for; `stream` waits for that
// stream at the end of the step.
ebd_status ebd_step_host(ebd_handle* h, const ebd_step_args* a, void* stream) {
  NvtxRange nvtx("ebd_step_host");
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  if (a == nullptr) return fail(h, EBD_ERR_INVALID_ARG, "args is NULL");
  if (a->batch < 0 || a->batch > h->cfg.max_batch || a->rows < 0 || a->rows > h->cfg.max_rows)
    return fail(h, EBD_ERR_INVALID_ARG, "batch/rows out of range");
  if (!a->cu_rows || !a->prefix_len || !a->row_pos || !a->hidden || !a->tokens || !a->mask ||
      !a->in_block || !a->blk_meta || !a->w_lm)
    return fail(h, EBD_ERR_INVALID_ARG, "missing host input");
  const bool attn = a->attn_out != nullptr;
  const bool kv = attn || a->kv_append;  // the window K/V feed the attention and the append
  if ((attn && !a->q) || (kv && (!a->k_win || !a->v_win)))
    return fail(h, EBD_ERR_INVALID_ARG, "missing host input (q / window K/V)");
  if (h->w_emb == nullptr) return fail(h, EBD_ERR_STATE, "bind the token embedding first");
  if (a->rows == 0 || a->batch == 0) return EBD_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const ebd_config& c = h->cfg;
  const size_t R = a->rows, B = a->batch, RM = c.max_rows, BM = c.max_batch;
  const size_t d = c.d_model, Hq = c.n_heads_q, Hkv = c.n_heads_kv, D = c.head_dim;
  uint8_t* p = h->staging;
  auto take = [&](size_t n) {
    uint8_t* q = p;
    p += (n + 255) / 256 * 256;
    return q;
  };
  ebd_step_args g = *a;
  int32_t* cu = reinterpret_cast<int32_t*>(take((BM + 1) * 4));
  int32_t* pl = reinterpret_cast<int32_t*>(take(BM * 4));
  int32_t* rp = reinterpret_cast<int32_t*>(take(RM * 4));
  uint16_t* hid = reinterpret_cast<uint16_t*>(take(RM * d * 2));
  uint16_t* q = reinterpret_cast<uint16_t*>(take(RM * Hq * D * 2));
  uint16_t* kw = reinterpret_cast<uint16_t*>(take(RM * Hkv * D * 2));
  uint16_t* vw = reinterpret_cast<uint16_t*>(take(RM * Hkv * D * 2));
  int32_t* tok = reinterpret_cast<int32_t*>(take(RM * 4));
  uint8_t* msk = take(RM);
  uint8_t* ib = take(RM);
  int32_t* meta = reinterpret_cast<int32_t*>(take(BM * 8));
  float* ao = reinterpret_cast<float*>(take(RM * Hq * D * 4));
  float* f[6];
  for (int i = 0; i < 6; ++i) f[i] = reinterpret_cast<float*>(take(RM * 4));
  int32_t* am = reinterpret_cast<int32_t*>(take(RM * 4));
  uint8_t* acc = take(RM);
  int32_t* sfx = reinterpret_cast<int32_t*>(take(BM * 8));
  const bool route = !seq_mode(h);
  // while `stream` is being captured into a graph the attention's inputs go
  // with the others (one capture-safe path; replays take it too)
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cap) != cudaSuccess) (void)cudaGetLastError();
  const bool dma = route && attn && cap == cudaStreamCaptureStatusNone && copy_route_ready(h);
  HostMover in{st, true};
  in.add(hid, a->hidden, R * d * 2);
  in.add(cu, a->cu_rows, (B + 1) * 4);
  in.add(pl, a->prefix_len, B * 4);
  in.add(rp, a->row_pos, R * 4);
  in.add(tok, a->tokens, R * 4);
  in.add(msk, a->mask, R);
  in.add(ib, a->in_block, R);
  in.add(meta, a->blk_meta, B * 8);
  if (a->suffix) in.add(sfx, a->suffix, B * 8);
  if (!dma) {
    if (attn) in.add(q, a->q, R * Hq * D * 2);
    if (kv) {
      in.add(kw, a->k_win, R * Hkv * D * 2);
      in.add(vw, a->v_win, R * Hkv * D * 2);
    }
  }
  // the copy stream forks before the gather, so that the LM head can be a
  // programmatic dependent of the gather kernel (it prefetches its first W
  // stages while the hidden rows come in)
  if (dma) {
    cudaError_t e0 = cudaEventRecord(h->ev_fork, st);
    if (e0 != cudaSuccess) return cuda_fail(h, e0, "copy stream event");
  }
  const bool gathered = in.list.n > 0;  // flush() launches the gather kernel
  cudaError_t e = in.flush();
  if (e != cudaSuccess) return cuda_fail(h, e, "host-to-device copy");
  unsigned ticket = 0;
  if (dma) {
    if (++h->ticket == 0) h->ticket = 1;  // 0 is the word's initial value
    ticket = h->ticket;
    const cudaMemcpyKind k = cudaMemcpyHostToDevice;
    if ((e = cudaStreamWaitEvent(h->s_copy, h->ev_fork, 0)) != cudaSuccess ||
        (e = cudaMemcpyAsync(q, a->q, R * Hq * D * 2, k, h->s_copy)) != cudaSuccess ||
        (e = cudaMemcpyAsync(kw, a->k_win, R * Hkv * D * 2, k, h->s_copy)) != cudaSuccess ||
        (e = cudaMemcpyAsync(vw, a->v_win, R * Hkv * D * 2, k, h->s_copy)) != cudaSuccess)
      return cuda_fail(h, e, "host-to-device copy (copy stream)");
    if (get_write_value()(reinterpret_cast<CUstream>(h->s_copy), reinterpret_cast<CUdeviceptr>(h->d_ready),
                          ticket, 0) != CUDA_SUCCESS)
      return fail(h, EBD_ERR_CUDA, "cuStreamWriteValue32 failed");
    if ((e = cudaEventRecord(h->ev_join, h->s_copy)) != cudaSuccess)
      return cuda_fail(h, e, "copy stream event");
  }
  g.cu_rows = cu; g.prefix_len = pl; g.row_pos = rp; g.hidden = hid;
  g.q = attn ? q : nullptr; g.k_win = kv ? kw : nullptr; g.v_win = kv ? vw : nullptr;
  g.tokens = tok; g.mask = msk; g.in_block = ib; g.blk_meta = meta;
  g.suffix = a->suffix ? sfx : nullptr;
  // A result buffer: the caller's own (its device address) where it is
  // mapped and aligned as the kernel's stores need, else the staging buffer,
  // copied back after the step.
  struct Back {
    void* host;
    const void* stage;
    size_t bytes;
  } back[16];
  int nback = 0;
  auto result = [&](void* host, void* stage, size_t bytes, uintptr_t align) -> void* {
    if (host == nullptr) return nullptr;
    if (route) {
      const void* dev = mapped_host(host);
      if (dev != nullptr && (reinterpret_cast<uintptr_t>(dev) & (align - 1)) == 0) return const_cast<void*>(dev);
    }
    back[nback++] = Back{host, stage, bytes};
    return stage;
  };
  StepRoute rt{gathered, dma ? h->d_ready : nullptr, ticket, nullptr, nullptr, nullptr, nullptr};
  rt.tokens_out = static_cast<int32_t*>(result(a->tokens, tok, R * 4, 4));
  rt.mask_out = static_cast<uint8_t*>(result(a->mask, msk, R, 1));
  rt.in_block_out = static_cast<uint8_t*>(result(a->in_block, ib, R, 1));
  rt.blk_meta_out = static_cast<int32_t*>(result(a->blk_meta, meta, B * 8, 4));
  g.attn_out = attn ? static_cast<float*>(result(a->attn_out, ao, R * Hq * D * 4, 16)) : nullptr;
  g.conf = static_cast<float*>(result(a->conf, f[0], R * 4, 4));
  g.entropy = static_cast<float*>(result(a->entropy, f[1], R * 4, 4));
  g.ent_norm = static_cast<float*>(result(a->ent_norm, f[2], R * 4, 4));
  g.gap = static_cast<float*>(result(a->gap, f[3], R * 4, 4));
  g.lbs_logit = static_cast<float*>(result(a->lbs_logit, f[4], R * 4, 4));
  g.lps_prob = static_cast<float*>(result(a->lps_prob, f[5], R * 4, 4));
  g.argmax = static_cast<int32_t*>(result(a->argmax, am, R * 4, 4));
  g.accepted = static_cast<uint8_t*>(result(a->accepted, acc, R, 1));
  if (route) {
    if ((s = check_args(h, &g, attn, true, true)) != EBD_OK) return s;
    (void)cudaGetLastError();  // a stale error of an earlier unrelated call is not ours
    s = step_run(h, &g, st, &rt);
  } else {
    s = ebd_step(h, &g, stream);  // in place on the staged decode state
  }
  if (dma) {  // later work on `stream` follows the copy stream too (also after a failed launch)
    if ((e = cudaStreamWaitEvent(st, h->ev_join, 0)) != cudaSuccess && s == EBD_OK)
      return cuda_fail(h, e, "copy stream join");
  }
  if (s != EBD_OK) return s;
  HostMover out{st, false};
  for (int i = 0; i < nback; ++i) out.add(back[i].host, back[i].stage, back[i].bytes);
  if ((e = out.flush()) != cudaSuccess) return cuda_fail(h, e, "device-to-host copy");
  return EBD_OK;
}

ebd_status ebd_profile_enable(ebd_handle* h, int mode) {
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  if (mode < 0 || mode > 2) return fail(h, EBD_ERR_INVALID_ARG, "profile mode must be 0, 1 or 2");
  h->profile = mode;
  return EBD_OK;
}

ebd_status ebd_profile_read(ebd_handle* h, float* ms) {
  if (h == nullptr || ms == nullptr) return EBD_ERR_INVALID_ARG;
  if (h->prof_mode == 0) return fail(h, EBD_ERR_STATE, "no profiled ebd_step recorded");
  cudaError_t e = cudaEventSynchronize(h->ev[3]);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaEventSynchronize");
  auto span = [&](int i, int j, float* out) { return cudaEventElapsedTime(out, h->ev[i], h->ev[j]); };
  if ((e = span(0, 1, &ms[1])) != cudaSuccess) return cuda_fail(h, e, "cudaEventElapsedTime");
  if (h->prof_mode == 1) {
    if ((e = span(1, 2, &ms[2])) != cudaSuccess) return cuda_fail(h, e, "cudaEventElapsedTime");
    if ((e = span(2, 3, &ms[0])) != cudaSuccess) return cuda_fail(h, e, "cudaEventElapsedTime");
    if (!h->prof_attn) ms[0] = 0.f;
  } else {
    if ((e = span(1, 3, &ms[2])) != cudaSuccess) return cuda_fail(h, e, "cudaEventElapsedTime");
    ms[0] = -1.f;
  }
  return EBD_OK;
}

ebd_status ebd_sync_status(ebd_handle* h, void* stream) {
  if (h == nullptr) return EBD_ERR_INVALID_ARG;
  ebd_status s = check_device(h);
  if (s != EBD_OK) return s;
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "stream synchronize");
  int v = 0;
  if ((e = cudaMemcpy(&v, h->d_status, sizeof(int), cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(h, e, "status read");
  if (v != 0) {
    cudaMemset(h->d_status, 0, sizeof(int));
    const int slots = h->cfg.max_batch * h->cfg.n_heads_kv * h->attn_max_qtiles;
    if (h->tickets) cudaMemset(h->tickets, 0, static_cast<size_t>(slots) * sizeof(int));
    cudaDeviceSynchronize();
    h->err = "device reported status " + std::to_string(v);
  }
  return v;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free LM-head statistics (ebd_lm_stats_noalloc).
//
// The paper has no counterpart: this serves callers that must not allocate
// device memory when they ask for the statistics of step 2.  Two kinds:
//   - a serving process whose weight and KV-cache pools reserved the free HBM
//     up front, where any further cudaMalloc fails or fragments the pool;
//   - a decode loop that must not stall, where cudaFree (and cudaMalloc on
//     some paths) synchronises the whole device.
// The handle path allocates its workspace in ebd_create; this path needs no
// handle: the LM-head partials live in the file-scope array below, sized for
// EBD_NOALLOC_MAX_ROWS rows x EBD_NOALLOC_MAX_PARTS partials per row
// (64 x 160 x 20 bytes = 200 KiB).  Nothing in it has to start at zero: every
// LM-head CTA writes its partial of every row before the merge reads it.
// There is one copy per device, so calls that overlap in time on one device
// (two streams, or two host threads) race on it; calls on one stream are
// ordered and safe.
// ---------------------------------------------------------------------------
static __device__ __align__(256) unsigned char
    g_noalloc_scratch[static_cast<size_t>(EBD_NOALLOC_MAX_ROWS) * EBD_NOALLOC_MAX_PARTS *
                      (sizeof(float4) + sizeof(int))];

namespace {

constexpr int kNoAllocMaxDevices = 64;
struct NoAllocDevice {
  bool ready = false;
  int num_sms = 0;
  float4* part_f = nullptr;  // [rows][grid], grid <= EBD_NOALLOC_MAX_PARTS
  int* part_i = nullptr;     // [rows][grid]
};
NoAllocDevice g_noalloc_dev[kNoAllocMaxDevices];
std::mutex g_noalloc_mu;

// One-time setup of device `dev` (the current device): the scratch address
// (cudaGetSymbolAddress), the LM-head kernel attributes and the SM count.
// Allocates nothing.
ebd_status noalloc_setup(int dev, NoAllocDevice** out) {
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  NoAllocDevice& d = g_noalloc_dev[dev];
  if (!d.ready) {
    int major = 0, minor = 0, sms = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return EBD_ERR_CUDA;
    if (major != 10 || minor != 3) return EBD_ERR_UNSUPPORTED;
    void* base = nullptr;
    if (cudaGetSymbolAddress(&base, g_noalloc_scratch) != cudaSuccess) return EBD_ERR_CUDA;
    if (lm_configure() != cudaSuccess) return EBD_ERR_CUDA;
    d.num_sms = sms;
    d.part_f = static_cast<float4*>(base);
    d.part_i = reinterpret_cast<int*>(static_cast<unsigned char*>(base) +
                                      static_cast<size_t>(EBD_NOALLOC_MAX_ROWS) *
                                          EBD_NOALLOC_MAX_PARTS * sizeof(float4));
    d.ready = true;
  }
  *out = &d;
  return EBD_OK;
}

}  // namespace

extern "C" ebd_status ebd_lm_stats_noalloc(const uint16_t* hidden, const uint16_t* w_lm,
                                           int32_t w_lm_layout, int32_t rows, int32_t d_model,
                                           int32_t vocab, float* conf, float* entropy,
                                           float* ent_norm, float* gap, int32_t* argmax,
                                           int32_t* status, void* stream) {
  if (rows < 0 || d_model <= 0 || d_model % 8 || vocab < 2 || (w_lm_layout != 0 && w_lm_layout != 1))
    return EBD_ERR_INVALID_ARG;
  if (rows > EBD_NOALLOC_MAX_ROWS) return EBD_ERR_UNSUPPORTED;
  if (rows == 0) return EBD_OK;
  if (hidden == nullptr || w_lm == nullptr || status == nullptr ||
      reinterpret_cast<uintptr_t>(hidden) % 16 || reinterpret_cast<uintptr_t>(w_lm) % 16)
    return EBD_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EBD_ERR_CUDA;
  if (dev < 0 || dev >= kNoAllocMaxDevices) return EBD_ERR_UNSUPPORTED;
  NoAllocDevice* nd = nullptr;
  ebd_status s = noalloc_setup(dev, &nd);
  if (s != EBD_OK) return s;
  const bool packed = w_lm_layout == 1;
  const uint64_t units = (static_cast<uint64_t>(vocab) + kUnit - 1) / kUnit;
  const uint64_t nkb = (static_cast<uint64_t>(d_model) + 63) / 64;
  CUtensorMap tw, th;
  (void)units;
  (void)nkb;
  if (!encode_w_lm(&tw, w_lm, vocab, d_model, packed, 0)) return EBD_ERR_CUDA;
  LmParams p{};
  lm_plan(p, rows, vocab, d_model,
          nd->num_sms < EBD_NOALLOC_MAX_PARTS ? nd->num_sms : EBD_NOALLOC_MAX_PARTS);
  if (p.stages < 2 || p.grid > EBD_NOALLOC_MAX_PARTS) return EBD_ERR_UNSUPPORTED;
  p.row0 = 0;
  p.part_rows = EBD_NOALLOC_MAX_ROWS;
  p.packed = packed ? 1 : 0;
  p.part_f = nd->part_f;
  p.part_i = nd->part_i;
  p.status = status;
  p.limit_ns = kLimitNs;
  p.force_timeout = 0;
  {
    const uint64_t dims[2] = {static_cast<uint64_t>(d_model), static_cast<uint64_t>(rows)};
    const uint64_t str[1] = {static_cast<uint64_t>(d_model) * 2};
    const uint32_t box[2] = {64, static_cast<uint32_t>(p.nb)};
    if (!encode_bf16(&th, hidden, 2, dims, str, box)) return EBD_ERR_CUDA;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (launch_lm_stats(tw, th, p, st) != cudaSuccess) return EBD_ERR_CUDA;
  const float inv = static_cast<float>(1.0 / std::log(static_cast<double>(vocab)));
  if (launch_merge_stats(nd->part_f, nd->part_i, rows, p.grid, vocab, inv, conf, entropy, ent_norm,
                         gap, argmax, status, st) != cudaSuccess)
    return EBD_ERR_CUDA;
  return EBD_OK;
}
