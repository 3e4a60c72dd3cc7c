// C ABI of the CORA-Diff library: model and session objects, the per-step
// CUDA graph (dense pass -> active-row LM head + Eq. 1 -> gate), the decode
// loop, and the standalone kernel entry points.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/cora.h"
#include "cora_kernels.h"

// ------------------------------------------------------------------ errors
static thread_local std::string g_last_error;

static int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return code;
}

// Records `msg` as the calling thread's last error and returns `code`
// (for entry points implemented in other translation units).
int cora_set_error(int code, const char* msg) {
  g_last_error = msg;
  return code;
}

#define CK(call)                                                                        \
  do {                                                                                  \
    cudaError_t e_ = (call);                                                            \
    if (e_ != cudaSuccess) {                                                            \
      return fail(e_ == cudaErrorMemoryAllocation ? CORA_ENOMEM : CORA_ECUDA, "%s: %s", \
                  #call, cudaGetErrorString(e_));                                       \
    }                                                                                   \
  } while (0)

#define REQUIRE(cond, ...)                     \
  do {                                         \
    if (!(cond)) return fail(CORA_EINVAL, __VA_ARGS__); \
  } while (0)

extern "C" const char* cora_last_error(void) { return g_last_error.c_str(); }
extern "C" int cora_version(void) { return 200; }

// --------------------------------------------------------- device context
namespace {

struct DeviceCtx {
  bool ready = false;
  bool prepared = false;
  int num_sms = 0;
  int* err = nullptr;          // device error word for standalone ops
  void* scratch = nullptr;     // partials for standalone reductions
  size_t scratch_bytes = 0;
  GemmWorkspace gemm_ws{nullptr, nullptr};  // stream-K workspace for cora_op_gemm
  int* counters = nullptr;     // completion counters of the fused reductions
  size_t n_counters = 0;
};

std::mutex g_mu;
DeviceCtx g_dev[16];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

int device_ctx(DeviceCtx** out) {
  int dev = 0;
  CK(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 16) return fail(CORA_EINVAL, "device index %d unsupported", dev);
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceCtx& c = g_dev[dev];
  if (!c.ready) {
    CK(cudaDeviceGetAttribute(&c.num_sms, cudaDevAttrMultiProcessorCount, dev));
    CK(cudaMalloc(&c.err, sizeof(int)));
    CK(cudaMemset(c.err, 0, sizeof(int)));
    CK(cudaMalloc(&c.gemm_ws.partial, gemm_workspace_bytes(c.num_sms)));
    CK(cudaMalloc(&c.gemm_ws.flags, sizeof(int) * kGemmFlagCount));
    CK(cudaMemset(c.gemm_ws.flags, 0, sizeof(int) * kGemmFlagCount));
    if (!g_encode) {
      cudaDriverEntryPointQueryResult q;
      void* fn = nullptr;
      CK(cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q));
      if (q != cudaDriverEntryPointSuccess || !fn) return fail(CORA_ECUDA, "cuTensorMapEncodeTiled unavailable");
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    c.ready = true;
  }
  *out = &c;
  return CORA_OK;
}

int scratch_reserve(DeviceCtx* c, size_t bytes, void** out) {
  if (c->scratch_bytes < bytes) {
    if (c->scratch) CK(cudaFree(c->scratch));
    c->scratch = nullptr;
    c->scratch_bytes = 0;
    CK(cudaMalloc(&c->scratch, bytes));
    c->scratch_bytes = bytes;
  }
  *out = c->scratch;
  return CORA_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Partials [n_chunks, rows] (shared scratch) and n_groups completion
// counters (a separate allocation, zeroed when grown; every launch leaves the
// counters it used at zero).  Calls on one device are stream-ordered users of
// the same scratch.
int reduce_scratch(DeviceCtx* c, int n_chunks, int rows, int n_groups, Top1Part** parts, int** counters) {
  void* p = nullptr;
  int rc = scratch_reserve(c, size_t(n_chunks) * rows * sizeof(Top1Part), &p);
  if (rc) return rc;
  if (c->n_counters < size_t(n_groups)) {
    if (c->counters) CK(cudaFree(c->counters));
    c->counters = nullptr;
    c->n_counters = 0;
    CK(cudaMalloc(&c->counters, size_t(n_groups) * sizeof(int)));
    CK(cudaMemset(c->counters, 0, size_t(n_groups) * sizeof(int)));
    c->n_counters = size_t(n_groups);
  }
  *parts = static_cast<Top1Part*>(p);
  *counters = c->counters;
  return CORA_OK;
}

}  // namespace

bool make_tmap_2d(CUtensorMap* map, const void* base, int elem_bytes, uint64_t rows, uint64_t cols,
                  uint64_t row_stride_bytes, uint32_t box_rows, uint32_t box_cols) {
  if (!g_encode) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, elem_bytes == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                        const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_tmap_bf16_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t row_stride_bytes,
                       uint32_t box_rows, uint32_t box_cols) {
  return make_tmap_2d(map, base, 2, rows, cols, row_stride_bytes, box_rows, box_cols);
}

bool make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t stride1_bytes,
                       uint64_t stride2_bytes, uint32_t b0, uint32_t b1, uint32_t b2) {
  if (!g_encode) return false;
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  cuuint32_t box[3] = {b0, b1, b2};
  cuuint32_t estr[3] = {1, 1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Sets the shared-memory attributes of every kernel instance, once per device.
static int kernels_prepare() {
  DeviceCtx* dc = nullptr;
  int rc = device_ctx(&dc);
  if (rc) return rc;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!dc->prepared) {
    CK(gemm_prepare());
    CK(lm_head_prepare());
    CK(attention_tc_prepare());
    CK(attention_tc2_prepare());
    dc->prepared = true;
  }
  return CORA_OK;
}

// ------------------------------------------------------------------ model
struct cora_model {
  cora_model_config cfg{};
  int f_pad = 0;   // ffn rounded up to a multiple of 128
  int n_qkv = 0;   // (n_heads + 2 n_kv_heads) * head_dim
  int num_sms = 0;
  uint16_t* embed = nullptr;
  uint16_t* head = nullptr;
  uint16_t* final_norm = nullptr;
  std::vector<uint16_t*> attn_norm, ffn_norm, wqkv, wo, wgu, wdown;
  std::vector<CUtensorMap> tm_qkv, tm_o, tm_gu, tm_down;
  CUtensorMap tm_head{};
  std::vector<void*> allocs;
  cora_session* cached = nullptr;
};

static int model_alloc(cora_model* m, size_t bytes, uint16_t** out) {
  void* p = nullptr;
  CK(cudaMalloc(&p, bytes));
  m->allocs.push_back(p);
  *out = static_cast<uint16_t*>(p);
  return CORA_OK;
}

static void model_free(cora_model* m) {
  for (void* p : m->allocs) cudaFree(p);
  m->allocs.clear();
}

// Weight upload: [rows, cols] elements of `dtype` at src (row stride src_ld
// elements, "any" pointer) into bf16 dst (row stride dst_ld).  bf16 is copied
// as it is; fp32 is rounded to bf16 on the device, read in place when the
// caller's tensor is device-accessible, else through the staging buffer.
struct WeightUpload {
  int dtype = CORA_DTYPE_BF16;
  float* stage = nullptr;  // device staging buffer for fp32 host tensors
  size_t stage_elems = 0;
  ~WeightUpload() {
    if (stage) cudaFree(stage);
  }
};
constexpr size_t kStageBytes = size_t(256) << 20;

static size_t dtype_bytes(int dtype) { return dtype == CORA_DTYPE_F32 ? 4 : 2; }

static const void* elem_offset(const void* p, size_t elems, int dtype) {
  return static_cast<const char*>(p) + elems * dtype_bytes(dtype);
}

static int put_rows(WeightUpload& up, uint16_t* dst, size_t dst_ld, const void* src, size_t src_ld, size_t rows,
                    size_t cols) {
  if (up.dtype == CORA_DTYPE_BF16) {
    CK(cudaMemcpy2D(dst, dst_ld * 2, src, src_ld * 2, cols * 2, rows, cudaMemcpyDefault));
    return CORA_OK;
  }
  cudaPointerAttributes at{};
  CK(cudaPointerGetAttributes(&at, src));
  if (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged) {
    launch_f32_to_bf16_2d(static_cast<const float*>(src), int64_t(src_ld), dst, int64_t(dst_ld), int64_t(rows),
                          int64_t(cols), nullptr);
    CK(cudaGetLastError());
    CK(cudaDeviceSynchronize());
    return CORA_OK;
  }
  if (!up.stage) {
    up.stage_elems = kStageBytes / 4;
    CK(cudaMalloc(&up.stage, up.stage_elems * 4));
  }
  const size_t rows_per_chunk = std::max<size_t>(1, up.stage_elems / cols);
  for (size_t r0 = 0; r0 < rows; r0 += rows_per_chunk) {
    const size_t n = std::min(rows_per_chunk, rows - r0);
    CK(cudaMemcpy2D(up.stage, cols * 4, elem_offset(src, r0 * src_ld, CORA_DTYPE_F32), src_ld * 4, cols * 4, n,
                    cudaMemcpyHostToDevice));
    launch_f32_to_bf16_2d(up.stage, int64_t(cols), dst + r0 * dst_ld, int64_t(dst_ld), int64_t(n), int64_t(cols),
                          nullptr);
    CK(cudaGetLastError());
    CK(cudaDeviceSynchronize());  // the staging buffer is reused by the next chunk
  }
  return CORA_OK;
}

static int copy_rows(WeightUpload& up, uint16_t* dst, const void* src, size_t rows, size_t cols) {
  return put_rows(up, dst, cols, src, cols, rows, cols);
}

extern "C" int cora_model_destroy(cora_model* m);
extern "C" int cora_session_destroy(cora_session* s);

extern "C" int cora_model_create(const cora_model_config* cfg, const cora_weights* w, cora_model** out) {
  REQUIRE(cfg && w && out, "cora_model_create: NULL argument");
  const cora_model_config c = *cfg;
  REQUIRE(c.n_layers >= 1 && c.d_model >= 128 && c.d_model % 128 == 0, "d_model must be a positive multiple of 128");
  REQUIRE(c.head_dim == 64 || c.head_dim == 128, "head_dim must be 64 or 128");
  REQUIRE(c.n_heads >= 1 && c.n_kv_heads >= 1 && c.n_heads % c.n_kv_heads == 0, "n_heads %% n_kv_heads != 0");
  REQUIRE((c.n_heads * c.head_dim) % 64 == 0, "n_heads * head_dim must be a multiple of 64");
  REQUIRE(((c.n_heads + 2 * c.n_kv_heads) * c.head_dim) % 128 == 0,
          "(n_heads + 2 n_kv_heads) * head_dim must be a multiple of 128");
  REQUIRE(c.ffn >= 1 && c.vocab >= 2 && c.mask_id >= 0 && c.mask_id < c.vocab, "bad ffn/vocab/mask_id");
  REQUIRE(c.norm_eps >= 0.f && c.rope_theta > 0.f, "bad norm_eps/rope_theta");
  REQUIRE(w->dtype == CORA_DTYPE_BF16 || w->dtype == CORA_DTYPE_F32, "cora_model_create: unknown weight dtype %d",
          w->dtype);
  REQUIRE(w->embed && w->lm_head && w->wq && w->wk && w->wv && w->wo && w->w_gate && w->w_up && w->w_down,
          "cora_model_create: NULL weight");
  for (int l = 0; l < c.n_layers; ++l)
    REQUIRE(w->wq[l] && w->wk[l] && w->wv[l] && w->wo[l] && w->w_gate[l] && w->w_up[l] && w->w_down[l],
            "cora_model_create: NULL weight in layer %d", l);

  DeviceCtx* dc = nullptr;
  int rc = device_ctx(&dc);
  if (rc) return rc;
  if ((rc = kernels_prepare())) return rc;

  cora_model* m = new cora_model();
  m->cfg = c;
  m->num_sms = dc->num_sms;
  m->f_pad = (c.ffn + 127) / 128 * 128;
  m->n_qkv = (c.n_heads + 2 * c.n_kv_heads) * c.head_dim;
  const size_t d = c.d_model, hq = size_t(c.n_heads) * c.head_dim, hkv = size_t(c.n_kv_heads) * c.head_dim;
  const size_t F = c.ffn, FP = m->f_pad;

#define MK(call)          \
  do {                    \
    int r_ = (call);      \
    if (r_) {             \
      cora_model_destroy(m); \
      return r_;          \
    }                     \
  } while (0)

  WeightUpload up;
  up.dtype = w->dtype;
  const int dt = w->dtype;
  MK(model_alloc(m, size_t(c.vocab) * d * 2, &m->embed));
  MK(copy_rows(up, m->embed, w->embed, c.vocab, d));
  MK(model_alloc(m, size_t(c.vocab) * d * 2, &m->head));
  MK(copy_rows(up, m->head, w->lm_head, c.vocab, d));
  if (w->final_norm) {
    MK(model_alloc(m, d * 2, &m->final_norm));
    MK(copy_rows(up, m->final_norm, w->final_norm, 1, d));
  }
  for (int l = 0; l < c.n_layers; ++l) {
    uint16_t *an = nullptr, *fn = nullptr, *qkv, *wo, *gu, *dn;
    if (w->attn_norm && w->attn_norm[l]) {
      MK(model_alloc(m, d * 2, &an));
      MK(copy_rows(up, an, w->attn_norm[l], 1, d));
    }
    if (w->ffn_norm && w->ffn_norm[l]) {
      MK(model_alloc(m, d * 2, &fn));
      MK(copy_rows(up, fn, w->ffn_norm[l], 1, d));
    }
    MK(model_alloc(m, size_t(m->n_qkv) * d * 2, &qkv));
    MK(copy_rows(up, qkv, w->wq[l], hq, d));
    MK(copy_rows(up, qkv + hq * d, w->wk[l], hkv, d));
    MK(copy_rows(up, qkv + (hq + hkv) * d, w->wv[l], hkv, d));
    MK(model_alloc(m, d * hq * 2, &wo));
    MK(copy_rows(up, wo, w->wo[l], d, hq));
    // gate/up interleaved in groups of 128 rows: [gate 128 | up 128] per group.
    MK(model_alloc(m, 2 * FP * d * 2, &gu));
    if (FP != F) CK(cudaMemset(gu, 0, 2 * FP * d * 2));
    for (size_t g0 = 0; g0 < F; g0 += 128) {
      const size_t n = (F - g0) < 128 ? (F - g0) : 128;
      MK(copy_rows(up, gu + (2 * g0) * d, elem_offset(w->w_gate[l], g0 * d, dt), n, d));
      MK(copy_rows(up, gu + (2 * g0 + 128) * d, elem_offset(w->w_up[l], g0 * d, dt), n, d));
    }
    MK(model_alloc(m, d * FP * 2, &dn));
    if (FP != F) CK(cudaMemset(dn, 0, d * FP * 2));
    MK(put_rows(up, dn, FP, w->w_down[l], F, d, F));
    m->attn_norm.push_back(an);
    m->ffn_norm.push_back(fn);
    m->wqkv.push_back(qkv);
    m->wo.push_back(wo);
    m->wgu.push_back(gu);
    m->wdown.push_back(dn);
    CUtensorMap t1, t2, t3, t4;
    // Weight (B operand) maps use 128-row boxes for every GEMM kernel.
    bool ok = make_tmap_bf16_2d(&t1, qkv, m->n_qkv, d, d * 2, 128, 64) &&
              make_tmap_bf16_2d(&t2, wo, d, hq, hq * 2, 128, 64) &&
              make_tmap_bf16_2d(&t3, gu, 2 * FP, d, d * 2, 128, 64) &&
              make_tmap_bf16_2d(&t4, dn, d, FP, FP * 2, 128, 64);
    if (!ok) {
      cora_model_destroy(m);
      return fail(CORA_ECUDA, "tensor map encoding failed (layer %d)", l);
    }
    m->tm_qkv.push_back(t1);
    m->tm_o.push_back(t2);
    m->tm_gu.push_back(t3);
    m->tm_down.push_back(t4);
  }
  if (!make_tmap_bf16_2d(&m->tm_head, m->head, c.vocab, d, d * 2, 128, 64)) {
    cora_model_destroy(m);
    return fail(CORA_ECUDA, "tensor map encoding failed (lm head)");
  }
#undef MK
  CK(cudaDeviceSynchronize());
  *out = m;
  return CORA_OK;
}

// ---------------------------------------------------------------- session
struct cora_session {
  cora_model* m = nullptr;
  int B = 0, P = 0, G = 0, S = 0, BL = 0, T = 0, n_blocks = 0, M = 0, R = 0;
  float tau = 0.f;
  cora_decode_options opt{CORA_SCHEDULE_FIXED, CORA_PERSIST_BLOCK, -1, CORA_CACHE_NONE};
  int K = 0;
  cudaStream_t stream = nullptr;
  std::vector<void*> allocs;
  int32_t* prompt = nullptr;   // [B, P] copy used by reset
  int32_t* tokens = nullptr;   // [B, S]
  float* h = nullptr;          // [M, d] residual stream
  uint16_t* xn = nullptr;      // [M, d] normalised activations
  uint16_t* qkv = nullptr;     // [M, n_qkv]
  uint16_t* attn = nullptr;    // [M, Hq*hd]
  uint16_t* act = nullptr;     // [M, f_pad]
  uint16_t* xf = nullptr;      // [R, d] final-normed active rows
  float* rope = nullptr;       // [S, hd/2, 2]
  float* rope_t = nullptr;     // [hd/2, S, 2] (the same table, frequency-major)
  Top1Part* parts = nullptr;   // [n_parts, R]
  int n_parts = 0;
  int32_t* ctrl = nullptr;     // [B, 4]
  uint8_t* state = nullptr;    // [B, G]
  int32_t* persist = nullptr;  // [B, BL]
  int32_t* prev = nullptr;     // [B, BL]
  float* conf = nullptr;       // [B, BL]
  int32_t* argmax = nullptr;   // [B, BL]
  uint8_t* unmask = nullptr;   // [B, BL]
  uint8_t* accept = nullptr;   // [B, BL]
  uint8_t* blk_done = nullptr; // [B] block had no unresolved position after the last step
  int32_t* status = nullptr;   // device {all_done (byte 0), error word}
  int32_t* status_h = nullptr; // pinned host copy
  long long* diag = nullptr;   // [B][3] disagreement counts
  CUtensorMap tm_xn{}, tm_attn{}, tm_act{};
  // Eq. 1 rows: Re = B * rows_per_seq (rows_per_seq = BL, or G for carry-over
  // persistence), normalised into xf and run through the LM head in chunks
  // of chunk_rows rows, one tensor map each.
  int rows_per_seq = 0, Re = 0, chunk_rows = 0, n_chunks = 0;
  std::vector<CUtensorMap> tm_xf;
  CUtensorMap tmo_qkv{}, tmo_h{}, tmo_act{};  // GEMM output maps
  CUtensorMap tm_qkv_in{};                     // QKV as the attention kernel's TMA source
  GemmWorkspace gemm_ws{nullptr, nullptr};
  // Prefix-cache mode: per-layer QKV buffers hold every layer's keys/values
  // (written in full by a block's dense first pass, on the recomputed rows by
  // its later passes); one graph per block for the later passes.
  std::vector<uint16_t*> qkv_l;
  std::vector<CUtensorMap> tmo_qkv_l, tm_qkv_in_l, tmo_qkv3_l;
  std::vector<cudaGraphExec_t> cgraph;
  int32_t next_info = 1;                // status[3] of the last step: bit 0 dense pass next, bits 1.. block
  cudaGraphExec_t graph = nullptr;      // one step
  cudaGraphExec_t run_graph = nullptr;  // WHILE node around one step: a whole decode (null: not available)
  int32_t max_iters = 0;                // n_blocks * T
  int64_t batched_passes = 0;
  bool finished = false;
};

// One tensor map per LM-head chunk of the normalised Eq. 1 rows.
static bool make_xf_maps(cora_session* s, size_t d) {
  s->tm_xf.assign(size_t(s->n_chunks), CUtensorMap{});
  for (int ch = 0; ch < s->n_chunks; ++ch) {
    const int rows_c = std::min(s->chunk_rows, s->Re - ch * s->chunk_rows);
    if (!make_tmap_bf16_2d(&s->tm_xf[ch], s->xf + size_t(ch) * s->chunk_rows * d, rows_c, d, d * 2,
                           lm_head_npad(rows_c), 64))
      return false;
  }
  return true;
}

template <typename T>
static int sess_alloc(cora_session* s, size_t count, T** out) {
  void* p = nullptr;
  CK(cudaMalloc(&p, count * sizeof(T) < 16 ? 16 : count * sizeof(T)));
  s->allocs.push_back(p);
  *out = static_cast<T*>(p);
  return CORA_OK;
}

// Optional per-launch event recorder (profiling path only; the graph path
// passes nullptr).
struct LaunchRecorder {
  std::vector<cudaEvent_t> ev;
  std::vector<int32_t> kinds;
  cudaStream_t st = nullptr;
  int mark(int kind) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return -1;
    cudaEventRecord(e, st);
    ev.push_back(e);
    if (kind >= 0) kinds.push_back(kind);
    return 0;
  }
  ~LaunchRecorder() {
    for (auto e : ev) cudaEventDestroy(e);
  }
};

#define REC(kind) \
  if (rec) rec->mark(kind)

// One dense pass + Eq. 1 + gate.  With `loop`, the step is the body of the
// whole-decode WHILE node: the status read-back is replaced by the kernel
// that sets the loop condition.
static int enqueue_step(cora_session* s, LaunchRecorder* rec = nullptr,
                        const cudaGraphConditionalHandle* loop = nullptr, int cached_block = -1) {
  cora_model* m = s->m;
  const cora_model_config& c = m->cfg;
  const int d = c.d_model;
  // cached_block >= 0: a later pass of that block in prefix-cache mode, over
  // the packed rows lo .. S-1 of every sequence (Ls per sequence).
  const bool packed = cached_block >= 0;
  const bool cache = s->opt.cache == CORA_CACHE_PREFIX;
  const int lo = packed ? s->P + cached_block * s->BL : 0;
  const int Ls = s->S - lo;
  const int M = s->B * Ls;
  int* err = s->status + 1;
  cudaStream_t st = s->stream;
  if (rec) {
    rec->st = st;
    rec->mark(-1);
  }
  launch_embed(s->tokens, m->embed, s->h, M, d, s->S, lo, packed ? Ls : 0, st);
  REC(CORA_KIND_EMBED);
  for (int l = 0; l < c.n_layers; ++l) {
    launch_rmsnorm(s->h, m->attn_norm[l], s->xn, M, d, c.norm_eps, st);
    REC(CORA_KIND_RMSNORM);
    uint16_t* qkv = cache ? s->qkv_l[l] : s->qkv;
    GemmEpilogue e1{qkv, m->n_qkv, CORA_EPI_ROPE_BF16, s->rope, Ls, c.head_dim,
                    (c.n_heads + c.n_kv_heads) * c.head_dim, 1};
    e1.rope_pos0 = lo;
    e1.rope_t = s->rope_t;
    e1.rope_tn = s->S;
    e1.out3d = packed ? 1 : 0;
    e1.a_ptr = s->xn;
    e1.a_rows = s->M;
    e1.out_rows_per_seq = s->S;
    const CUtensorMap& tmo = packed ? s->tmo_qkv3_l[l] : cache ? s->tmo_qkv_l[l] : s->tmo_qkv;
    CK(launch_gemm(s->tm_xn, m->tm_qkv[l], tmo, M, m->n_qkv, d, e1, s->gemm_ws, err, m->num_sms, st));
    REC(CORA_KIND_GEMM_QKV);
    CK(launch_attention_tc(cache ? s->tm_qkv_in_l[l] : s->tm_qkv_in, s->attn, s->B, s->S, c.n_heads, c.n_kv_heads,
                           c.head_dim, lo, Ls, err, m->num_sms, st));
    REC(CORA_KIND_ATTENTION);
    GemmEpilogue e2{s->h, d, CORA_EPI_RESID_F32, nullptr, 0, 0, 0, 1};
    e2.a_ptr = s->attn;
    e2.a_rows = s->M;
    CK(launch_gemm(s->tm_attn, m->tm_o[l], s->tmo_h, M, d, c.n_heads * c.head_dim, e2, s->gemm_ws, err, m->num_sms,
                   st));
    REC(CORA_KIND_GEMM_O);
    launch_rmsnorm(s->h, m->ffn_norm[l], s->xn, M, d, c.norm_eps, st);
    REC(CORA_KIND_RMSNORM);
    GemmEpilogue e3{s->act, m->f_pad, CORA_EPI_SWIGLU, nullptr, 0, 0, 0, 1};
    e3.a_ptr = s->xn;
    e3.a_rows = s->M;
    CK(launch_gemm(s->tm_xn, m->tm_gu[l], s->tmo_act, M, 2 * m->f_pad, d, e3, s->gemm_ws, err, m->num_sms, st));
    REC(CORA_KIND_GEMM_GATE_UP);
    GemmEpilogue e4 = e2;  // residual epilogue, A = the SwiGLU output
    e4.a_ptr = s->act;
    CK(launch_gemm(s->tm_act, m->tm_down[l], s->tmo_h, M, d, m->f_pad, e4, s->gemm_ws, err, m->num_sms, st));
    REC(CORA_KIND_GEMM_DOWN);
  }
  launch_final_norm_rows(s->h, m->final_norm, s->ctrl, s->xf, s->B, packed ? Ls : s->S, packed ? -1 : s->P, s->BL,
                         s->n_blocks, d, c.norm_eps, s->rows_per_seq, st);
  REC(CORA_KIND_FINAL_NORM);
  for (int ch = 0; ch < s->n_chunks; ++ch) {
    const int rows_c = std::min(s->chunk_rows, s->Re - ch * s->chunk_rows);
    CK(launch_lm_head_top1(m->tm_head, s->tm_xf[ch], rows_c, c.vocab, d,
                           s->parts + size_t(ch) * s->n_parts * s->chunk_rows, s->n_parts, err, st));
    REC(CORA_KIND_LM_HEAD);
  }
  SessionGateArgs ga{s->parts, s->n_parts, s->ctrl,  s->tokens, s->state,  s->persist, s->prev,
                     s->conf,  s->argmax,  s->unmask, s->accept, reinterpret_cast<uint8_t*>(s->status),
                     s->blk_done, err,      s->B,       s->S,      s->P,      s->G,       s->BL,      s->T,
                     s->tau,   s->K,       s->opt.schedule, s->opt.eos_id, s->rows_per_seq, s->chunk_rows,
                     cache ? 1 : 0};
  launch_session_gate(ga, st);
  REC(CORA_KIND_GATE);
  CK(cudaGetLastError());
  if (loop)
    CK(launch_step_loop_cond(*loop, s->status, s->max_iters, st));
  else
    CK(cudaMemcpyAsync(s->status_h, s->status, (cache ? 4 : 2) * sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  return CORA_OK;
}

// The whole decode as one graph: a conditional WHILE node whose body is one
// step (captured into it), so no host round trip separates the passes.
// Returns false (and leaves no graph) where the runtime does not support it.
static bool build_run_graph(cora_session* s) {
  cudaGraph_t g = nullptr;
  if (cudaGraphCreate(&g, 0) != cudaSuccess) return false;
  bool ok = false;
  do {
    cudaGraphConditionalHandle h;
    if (cudaGraphConditionalHandleCreate(&h, g, 1, cudaGraphCondAssignDefault) != cudaSuccess) break;
    cudaGraphNodeParams p{};
    p.type = cudaGraphNodeTypeConditional;
    p.conditional.handle = h;
    p.conditional.type = cudaGraphCondTypeWhile;
    p.conditional.size = 1;
    cudaGraphNode_t node;
    if (cudaGraphAddNode(&node, g, nullptr, nullptr, 0, &p) != cudaSuccess) break;
    cudaGraph_t body = p.conditional.phGraph_out[0];
    if (cudaStreamBeginCaptureToGraph(s->stream, body, nullptr, nullptr, 0, cudaStreamCaptureModeThreadLocal) !=
        cudaSuccess)
      break;
    const int rc = enqueue_step(s, nullptr, &h);
    cudaGraph_t captured = nullptr;
    const cudaError_t ce = cudaStreamEndCapture(s->stream, &captured);
    if (rc != CORA_OK || ce != cudaSuccess) break;
    ok = cudaGraphInstantiate(&s->run_graph, g, 0) == cudaSuccess;
  } while (false);
  cudaGraphDestroy(g);
  if (!ok) {
    s->run_graph = nullptr;
    cudaGetLastError();  // the fallback is the host loop; clear the sticky-free error state
  }
  return ok;
}

extern "C" int cora_session_reset(cora_session* s, const int32_t* prompt) {
  REQUIRE(s, "cora_session_reset: NULL session");
  if (prompt && s->P > 0) CK(cudaMemcpyAsync(s->prompt, prompt, size_t(s->B) * s->P * 4, cudaMemcpyDefault, s->stream));
  launch_session_init(s->tokens, s->prompt, s->state, s->persist, s->prev, s->ctrl, s->status, s->B, s->P, s->S, s->G,
                      s->rows_per_seq, s->m->cfg.mask_id, s->stream);
  CK(cudaGetLastError());
  CK(cudaStreamSynchronize(s->stream));
  s->batched_passes = 0;
  s->next_info = 1;  // the first pass of block 0 is dense
  s->finished = false;
  return CORA_OK;
}

extern "C" int cora_session_create(cora_model* m, int32_t batch, const int32_t* prompt, int32_t prompt_len,
                                   int32_t gen_len, int32_t block_len, int32_t steps_per_block, float tau, int32_t K,
                                   cora_session** out) {
  return cora_session_create_ex(m, batch, prompt, prompt_len, gen_len, block_len, steps_per_block, tau, K, nullptr,
                                out);
}

extern "C" int cora_session_create_ex(cora_model* m, int32_t batch, const int32_t* prompt, int32_t prompt_len,
                                      int32_t gen_len, int32_t block_len, int32_t steps_per_block, float tau,
                                      int32_t K, const cora_decode_options* opt, cora_session** out) {
  REQUIRE(m && out, "cora_session_create: NULL argument");
  const cora_decode_options o = opt ? *opt : cora_decode_options{CORA_SCHEDULE_FIXED, CORA_PERSIST_BLOCK, -1, CORA_CACHE_NONE};
  REQUIRE(o.schedule == CORA_SCHEDULE_FIXED || o.schedule == CORA_SCHEDULE_REMAINING, "unknown schedule %d",
          o.schedule);
  REQUIRE(o.persistence == CORA_PERSIST_BLOCK || o.persistence == CORA_PERSIST_CARRY, "unknown persistence mode %d",
          o.persistence);
  REQUIRE(o.eos_id == -1 || (o.eos_id >= 0 && o.eos_id < m->cfg.vocab && o.eos_id != m->cfg.mask_id),
          "eos_id must be -1 or a vocabulary id other than the mask id");
  REQUIRE(o.cache == CORA_CACHE_NONE || o.cache == CORA_CACHE_PREFIX, "unknown cache mode %d", o.cache);
  REQUIRE(o.cache == CORA_CACHE_NONE || o.persistence == CORA_PERSIST_BLOCK,
          "the prefix cache is not combined with carry-over persistence");
  // Packed prefix-cache rows are stored in 32-row boxes that must not
  // straddle two sequences: every suffix length gen_len - b * block_len is
  // then a multiple of 32.
  REQUIRE(o.cache == CORA_CACHE_NONE || block_len == 32, "the prefix cache needs block_len == 32");
  REQUIRE(batch >= 1 && prompt_len >= 0 && gen_len >= 1, "bad batch/prompt_len/gen_len");
  REQUIRE(block_len >= 1 && block_len <= 32, "block_len must be in [1, 32]");
  REQUIRE(gen_len % block_len == 0, "gen_len %% block_len != 0");
  REQUIRE(steps_per_block >= 1, "steps_per_block must be >= 1");
  REQUIRE(batch * block_len <= 256, "batch * block_len must be <= 256");
  REQUIRE(prompt_len == 0 || prompt, "NULL prompt");
  const cora_model_config& c = m->cfg;
  cora_session* s = new cora_session();
  s->m = m;
  s->B = batch;
  s->P = prompt_len;
  s->G = gen_len;
  s->S = prompt_len + gen_len;
  s->BL = block_len;
  s->T = steps_per_block;
  s->n_blocks = gen_len / block_len;
  s->M = batch * s->S;
  s->R = batch * block_len;
  s->tau = tau;
  s->K = K;
  s->opt = o;
  s->rows_per_seq = o.persistence == CORA_PERSIST_CARRY ? gen_len : block_len;
  s->Re = batch * s->rows_per_seq;
  s->chunk_rows = std::min(s->Re, 256);
  s->n_chunks = (s->Re + s->chunk_rows - 1) / s->chunk_rows;
  const size_t d = c.d_model, M = s->M;
#define SK(call)              \
  do {                        \
    int r_ = (call);          \
    if (r_) {                 \
      cora_session_destroy(s); \
      return r_;              \
    }                         \
  } while (0)
  SK(cudaStreamCreateWithFlags(&s->stream, cudaStreamNonBlocking) == cudaSuccess ? 0
                                                                               : fail(CORA_ECUDA, "stream create"));
  SK(sess_alloc(s, size_t(batch) * (prompt_len > 0 ? prompt_len : 1), &s->prompt));
  SK(sess_alloc(s, M, &s->tokens));
  SK(sess_alloc(s, M * d, &s->h));
  SK(sess_alloc(s, M * d, &s->xn));
  SK(sess_alloc(s, M * size_t(m->n_qkv), &s->qkv));
  if (o.cache == CORA_CACHE_PREFIX) {
    for (int l = 0; l < c.n_layers; ++l) {
      uint16_t* q = nullptr;
      SK(sess_alloc(s, M * size_t(m->n_qkv), &q));
      s->qkv_l.push_back(q);
      CUtensorMap t_out, t_in, t_out3;
      if (!make_gemm_out_tmap(&t_out, q, int(M), m->n_qkv, CORA_EPI_ROPE_BF16) ||
          !make_tmap_bf16_2d(&t_in, q, M, size_t(m->n_qkv), size_t(m->n_qkv) * 2, 128, 64) ||
          !make_tmap_bf16_3d(&t_out3, q, size_t(m->n_qkv), size_t(s->S), size_t(batch), size_t(m->n_qkv) * 2,
                             size_t(s->S) * m->n_qkv * 2, 64, 32, 1))
        SK(fail(CORA_ECUDA, "tensor map encoding failed (prefix cache)"));
      s->tmo_qkv_l.push_back(t_out);
      s->tm_qkv_in_l.push_back(t_in);
      s->tmo_qkv3_l.push_back(t_out3);
    }
  }
  SK(sess_alloc(s, M * size_t(c.n_heads) * c.head_dim, &s->attn));
  SK(sess_alloc(s, M * size_t(m->f_pad), &s->act));
  SK(sess_alloc(s, size_t(s->Re) * d, &s->xf));
  SK(sess_alloc(s, size_t(s->S) * c.head_dim, &s->rope));
  SK(sess_alloc(s, size_t(s->S) * c.head_dim, &s->rope_t));
  s->n_parts = lm_head_parts_count(c.vocab, m->num_sms);
  SK(sess_alloc(s, size_t(s->n_parts) * s->n_chunks * s->chunk_rows, &s->parts));
  SK(sess_alloc(s, size_t(batch) * 4, &s->ctrl));
  SK(sess_alloc(s, size_t(batch) * gen_len, &s->state));
  SK(sess_alloc(s, size_t(s->Re), &s->persist));
  SK(sess_alloc(s, size_t(s->Re), &s->prev));
  SK(sess_alloc(s, size_t(s->Re), &s->conf));
  SK(sess_alloc(s, size_t(s->Re), &s->argmax));
  SK(sess_alloc(s, size_t(s->R), &s->unmask));
  SK(sess_alloc(s, size_t(s->R), &s->accept));
  SK(sess_alloc(s, size_t(batch), &s->blk_done));
  SK(sess_alloc(s, 4, &s->status));
  SK(sess_alloc(s, size_t(batch) * 3, &s->diag));
  SK(sess_alloc(s, gemm_workspace_bytes(m->num_sms) / sizeof(float), &s->gemm_ws.partial));
  SK(sess_alloc(s, size_t(kGemmFlagCount), &s->gemm_ws.flags));
  if (cudaMemset(s->gemm_ws.flags, 0, sizeof(int) * kGemmFlagCount) != cudaSuccess) SK(fail(CORA_ECUDA, "memset"));
  {
    void* hp = nullptr;
    if (cudaHostAlloc(&hp, 16, cudaHostAllocDefault) != cudaSuccess) SK(fail(CORA_ENOMEM, "pinned alloc"));
    s->status_h = static_cast<int32_t*>(hp);
  }
  // RoPE table in double precision on the host: angle = pos * theta^(-2j/hd).
  {
    const int half = c.head_dim / 2;
    std::vector<float> tab(size_t(s->S) * half * 2);
    for (int p = 0; p < s->S; ++p)
      for (int j = 0; j < half; ++j) {
        const double ang = double(p) * std::pow(double(c.rope_theta), -2.0 * j / c.head_dim);
        tab[(size_t(p) * half + j) * 2] = float(std::cos(ang));
        tab[(size_t(p) * half + j) * 2 + 1] = float(std::sin(ang));
      }
    std::vector<float> tab_t(tab.size());
    for (int p = 0; p < s->S; ++p)
      for (int j = 0; j < half; ++j)
        for (int e = 0; e < 2; ++e) tab_t[(size_t(j) * s->S + p) * 2 + e] = tab[(size_t(p) * half + j) * 2 + e];
    if (cudaMemcpy(s->rope, tab.data(), tab.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(s->rope_t, tab_t.data(), tab_t.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess)
      SK(fail(CORA_ECUDA, "rope table upload"));
  }
  const size_t hq = size_t(c.n_heads) * c.head_dim;
  bool ok = make_tmap_bf16_2d(&s->tm_xn, s->xn, M, d, d * 2, 128, 64) &&
            make_tmap_bf16_2d(&s->tm_attn, s->attn, M, hq, hq * 2, 128, 64) &&
            make_tmap_bf16_2d(&s->tm_act, s->act, M, m->f_pad, size_t(m->f_pad) * 2, 128, 64) &&
            make_xf_maps(s, d) &&
            make_gemm_out_tmap(&s->tmo_qkv, s->qkv, int(M), m->n_qkv, CORA_EPI_ROPE_BF16) &&
            make_tmap_bf16_2d(&s->tm_qkv_in, s->qkv, M, size_t(m->n_qkv), size_t(m->n_qkv) * 2, 128, 64) &&
            make_gemm_out_tmap(&s->tmo_h, s->h, int(M), int(d), CORA_EPI_RESID_F32) &&
            make_gemm_out_tmap(&s->tmo_act, s->act, int(M), m->f_pad, CORA_EPI_SWIGLU);
  if (!ok) SK(fail(CORA_ECUDA, "tensor map encoding failed (session)"));
  SK(cora_session_reset(s, prompt));
  // Capture one step (every launch, then the status read-back) as a graph.
  {
    cudaGraph_t g = nullptr;
    if (cudaStreamBeginCapture(s->stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
      SK(fail(CORA_ECUDA, "begin capture"));
    int rc = enqueue_step(s);
    cudaError_t ce = cudaStreamEndCapture(s->stream, &g);
    if (rc) {
      if (g) cudaGraphDestroy(g);
      SK(rc);
    }
    if (ce != cudaSuccess) SK(fail(CORA_ECUDA, "end capture: %s", cudaGetErrorString(ce)));
    ce = cudaGraphInstantiate(&s->graph, g, 0);
    cudaGraphDestroy(g);
    if (ce != cudaSuccess) SK(fail(CORA_ECUDA, "graph instantiate: %s", cudaGetErrorString(ce)));
  }
  s->max_iters = int32_t(s->n_blocks) * s->T;
  if (o.cache == CORA_CACHE_PREFIX) {
    // Later passes of block b: rows P + b * BL .. S-1 of every sequence.
    for (int b = 0; b < s->n_blocks; ++b) {
      cudaGraph_t g = nullptr;
      if (cudaStreamBeginCapture(s->stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
        SK(fail(CORA_ECUDA, "begin capture"));
      const int rc = enqueue_step(s, nullptr, nullptr, b);
      cudaError_t ce = cudaStreamEndCapture(s->stream, &g);
      if (rc) {
        if (g) cudaGraphDestroy(g);
        SK(rc);
      }
      if (ce != cudaSuccess) SK(fail(CORA_ECUDA, "end capture: %s", cudaGetErrorString(ce)));
      cudaGraphExec_t ge = nullptr;
      ce = cudaGraphInstantiate(&ge, g, 0);
      cudaGraphDestroy(g);
      if (ce != cudaSuccess) SK(fail(CORA_ECUDA, "graph instantiate: %s", cudaGetErrorString(ce)));
      s->cgraph.push_back(ge);
    }
  } else {
    build_run_graph(s);  // (the device loop runs one graph; prefix-cache sessions switch graphs on the host)
  }
#undef SK
  *out = s;
  return CORA_OK;
}

extern "C" int cora_session_destroy(cora_session* s) {
  if (!s) return CORA_OK;
  if (s->stream) cudaStreamSynchronize(s->stream);
  if (s->graph) cudaGraphExecDestroy(s->graph);
  if (s->run_graph) cudaGraphExecDestroy(s->run_graph);
  for (auto g : s->cgraph) cudaGraphExecDestroy(g);
  for (void* p : s->allocs) cudaFree(p);
  if (s->status_h) cudaFreeHost(s->status_h);
  if (s->stream) cudaStreamDestroy(s->stream);
  if (s->m && s->m->cached == s) s->m->cached = nullptr;
  delete s;
  return CORA_OK;
}

extern "C" int cora_model_destroy(cora_model* m) {
  if (!m) return CORA_OK;
  if (m->cached) cora_session_destroy(m->cached);
  model_free(m);
  delete m;
  return CORA_OK;
}

// One graph launch of the step at every unfinished sequence's own (block,
// step); waits for it and reads the status word.
static int step_once(cora_session* s, uint8_t* all_done_out) {
  if (s->finished) return fail(CORA_ESTATE, "every sequence has finished; reset the session");
  cudaGraphExec_t g = s->graph;
  if (!s->cgraph.empty() && !(s->next_info & 1)) {
    const int b = s->next_info >> 1;
    REQUIRE(b >= 0 && b < int(s->cgraph.size()), "prefix cache: bad block index %d", b);
    g = s->cgraph[size_t(b)];
  }
  CK(cudaGraphLaunch(g, s->stream));
  CK(cudaStreamSynchronize(s->stream));
  if (!s->cgraph.empty()) s->next_info = s->status_h[3];
  s->batched_passes += 1;
  const int32_t code = s->status_h[1];
  if (code != 0) return fail(CORA_ETIMEOUT, "device error word 0x%x after step", code);
  const uint8_t done = reinterpret_cast<const uint8_t*>(s->status_h)[0];
  s->finished = done != 0;
  if (all_done_out) *all_done_out = done;
  return CORA_OK;
}

extern "C" int cora_denoise_step(cora_session* s, int32_t block, int32_t step, float* conf_out, int32_t* argmax_out,
                                 uint8_t* done_out) {
  REQUIRE(s, "cora_denoise_step: NULL session");
  REQUIRE(block >= -1 && step >= -1, "cora_denoise_step: block and step must be >= 0, or -1 for no check");
  if (s->finished) return fail(CORA_ESTATE, "every sequence has finished; reset the session");
  if (block >= 0 || step >= 0) {
    std::vector<int32_t> ctrl(size_t(s->B) * 4);
    CK(cudaStreamSynchronize(s->stream));
    CK(cudaMemcpy(ctrl.data(), s->ctrl, ctrl.size() * 4, cudaMemcpyDeviceToHost));
    for (int b = 0; b < s->B; ++b) {
      const int32_t* c = &ctrl[size_t(b) * 4];
      if (c[3] || c[1] < 0) continue;  // finished, or waiting for the batch's next block (prefix cache)
      if ((block >= 0 && c[0] != block) || (step >= 0 && c[1] != step))
        return fail(CORA_ESTATE, "cora_denoise_step: sequence %d is at block %d step %d, not block %d step %d", b,
                    c[0], c[1], block, step);
    }
  }
  const int rc = step_once(s, nullptr);
  if (rc) return rc;
  if (conf_out) CK(cudaMemcpy(conf_out, s->conf, size_t(s->Re) * 4, cudaMemcpyDefault));
  if (argmax_out) CK(cudaMemcpy(argmax_out, s->argmax, size_t(s->Re) * 4, cudaMemcpyDefault));
  if (done_out) CK(cudaMemcpy(done_out, s->blk_done, size_t(s->B), cudaMemcpyDefault));
  return CORA_OK;
}

extern "C" int cora_session_finished(cora_session* s, uint8_t* finished_out) {
  REQUIRE(s && finished_out, "cora_session_finished: NULL argument");
  *finished_out = s->finished ? 1 : 0;
  return CORA_OK;
}

extern "C" int cora_session_run(cora_session* s, int32_t* steps_out, uint8_t* on_device_out) {
  REQUIRE(s, "cora_session_run: NULL session");
  if (s->finished) return fail(CORA_ESTATE, "every sequence has finished; reset the session");
  int32_t steps = 0;
  if (s->run_graph) {
    CK(cudaMemsetAsync(s->status + 2, 0, sizeof(int32_t), s->stream));
    CK(cudaGraphLaunch(s->run_graph, s->stream));
    CK(cudaMemcpyAsync(s->status_h, s->status, 3 * sizeof(int32_t), cudaMemcpyDeviceToHost, s->stream));
    CK(cudaStreamSynchronize(s->stream));
    steps = s->status_h[2];
    s->batched_passes += steps;
    if (s->status_h[1] != 0) return fail(CORA_ETIMEOUT, "device error word 0x%x after step", s->status_h[1]);
    s->finished = reinterpret_cast<const uint8_t*>(s->status_h)[0] != 0;
  } else {
    uint8_t done = 0;
    for (int32_t i = 0; i < s->max_iters && !done; ++i, ++steps) {
      const int rc = step_once(s, &done);
      if (rc) return rc;
    }
  }
  if (steps_out) *steps_out = steps;
  if (on_device_out) *on_device_out = s->run_graph ? 1 : 0;
  if (!s->finished) return fail(CORA_ESTATE, "decode did not finish within the horizon");
  return CORA_OK;
}

extern "C" int cora_session_disagreement(cora_session* s, cora_session* dense, int64_t* n_acc, int64_t* n_acc_diff,
                                         int64_t* n_out_diff) {
  REQUIRE(s && dense && n_acc && n_acc_diff && n_out_diff, "cora_session_disagreement: NULL argument");
  REQUIRE(s->B == dense->B && s->P == dense->P && s->G == dense->G, "the sessions' shapes differ");
  CK(cudaStreamSynchronize(dense->stream));
  launch_disagreement(s->tokens, s->state, dense->tokens, s->B, s->S, s->P, s->G, s->diag, s->stream);
  CK(cudaGetLastError());
  std::vector<long long> h(size_t(s->B) * 3);
  CK(cudaMemcpyAsync(h.data(), s->diag, h.size() * sizeof(long long), cudaMemcpyDeviceToHost, s->stream));
  CK(cudaStreamSynchronize(s->stream));
  for (int b = 0; b < s->B; ++b) {
    n_acc[b] = h[size_t(b) * 3];
    n_acc_diff[b] = h[size_t(b) * 3 + 1];
    n_out_diff[b] = h[size_t(b) * 3 + 2];
  }
  return CORA_OK;
}

extern "C" int cora_session_profile_step(cora_session* s, int32_t capacity, int32_t* kinds, float* ms,
                                         int32_t* n_out) {
  REQUIRE(s && kinds && ms && n_out, "cora_session_profile_step: NULL argument");
  if (s->finished) return fail(CORA_ESTATE, "every sequence has finished; reset the session");
  const int need = 3 + 7 * s->m->cfg.n_layers + 1;
  REQUIRE(capacity >= need, "cora_session_profile_step: capacity %d < %d launches", capacity, need);
  CK(cudaStreamSynchronize(s->stream));
  LaunchRecorder rec;
  // The pass the next cora_denoise_step would run: in a prefix-cache session
  // a later pass of the current block covers the rows from it on.
  const int cached_block = (!s->cgraph.empty() && !(s->next_info & 1)) ? (s->next_info >> 1) : -1;
  int rc = enqueue_step(s, &rec, nullptr, cached_block);
  if (rc) return rc;
  CK(cudaStreamSynchronize(s->stream));
  if (!s->cgraph.empty()) s->next_info = s->status_h[3];
  s->batched_passes += 1;
  const int n = static_cast<int>(rec.kinds.size());
  for (int i = 0; i < n; ++i) {
    float t = 0.f;
    CK(cudaEventElapsedTime(&t, rec.ev[i], rec.ev[i + 1]));
    kinds[i] = rec.kinds[i];
    ms[i] = t;
  }
  *n_out = n;
  if (s->status_h[1] != 0) return fail(CORA_ETIMEOUT, "device error word 0x%x after step", s->status_h[1]);
  s->finished = reinterpret_cast<const uint8_t*>(s->status_h)[0] != 0;
  return CORA_OK;
}

extern "C" int cora_session_stream(cora_session* s, void** out) {
  REQUIRE(s && out, "NULL argument");
  *out = static_cast<void*>(s->stream);
  return CORA_OK;
}

extern "C" int cora_session_batched_passes(cora_session* s, int64_t* out) {
  REQUIRE(s && out, "NULL argument");
  *out = s->batched_passes;
  return CORA_OK;
}

extern "C" int cora_session_read(cora_session* s, int32_t* tokens, uint8_t* state, int32_t* persist, int32_t* prev,
                                 int32_t* ctrl, float* conf, int32_t* argmax, uint8_t* unmask, uint8_t* accept) {
  REQUIRE(s, "cora_session_read: NULL session");
  CK(cudaStreamSynchronize(s->stream));
  if (tokens) CK(cudaMemcpy(tokens, s->tokens, size_t(s->M) * 4, cudaMemcpyDeviceToHost));
  if (state) CK(cudaMemcpy(state, s->state, size_t(s->B) * s->G, cudaMemcpyDeviceToHost));
  if (persist) CK(cudaMemcpy(persist, s->persist, size_t(s->Re) * 4, cudaMemcpyDeviceToHost));
  if (prev) CK(cudaMemcpy(prev, s->prev, size_t(s->Re) * 4, cudaMemcpyDeviceToHost));
  if (ctrl) CK(cudaMemcpy(ctrl, s->ctrl, size_t(s->B) * 16, cudaMemcpyDeviceToHost));
  if (conf) CK(cudaMemcpy(conf, s->conf, size_t(s->Re) * 4, cudaMemcpyDeviceToHost));
  if (argmax) CK(cudaMemcpy(argmax, s->argmax, size_t(s->Re) * 4, cudaMemcpyDeviceToHost));
  if (unmask) CK(cudaMemcpy(unmask, s->unmask, size_t(s->R), cudaMemcpyDeviceToHost));
  if (accept) CK(cudaMemcpy(accept, s->accept, size_t(s->R), cudaMemcpyDeviceToHost));
  return CORA_OK;
}

extern "C" int cora_session_write(cora_session* s, const int32_t* tokens, const uint8_t* state, const int32_t* persist,
                                  const int32_t* prev, const int32_t* ctrl) {
  REQUIRE(s, "cora_session_write: NULL session");
  CK(cudaStreamSynchronize(s->stream));
  if (tokens) CK(cudaMemcpy(s->tokens, tokens, size_t(s->M) * 4, cudaMemcpyHostToDevice));
  if (state) CK(cudaMemcpy(s->state, state, size_t(s->B) * s->G, cudaMemcpyHostToDevice));
  if (persist) CK(cudaMemcpy(s->persist, persist, size_t(s->Re) * 4, cudaMemcpyHostToDevice));
  if (prev) CK(cudaMemcpy(s->prev, prev, size_t(s->Re) * 4, cudaMemcpyHostToDevice));
  if (ctrl) {
    CK(cudaMemcpy(s->ctrl, ctrl, size_t(s->B) * 16, cudaMemcpyHostToDevice));
    // Prefix cache: a canvas written at a block's first step (or at another
    // block) starts with that block's dense pass, which refreshes the kept
    // keys/values; a later step of the current block keeps them.
    const int32_t cur = s->next_info >> 1;
    s->next_info = (ctrl[1] == 0 || ctrl[0] != cur) ? (1 | (ctrl[0] << 1)) : (ctrl[0] << 1);
    bool all = true;
    for (int b = 0; b < s->B; ++b) all = all && ctrl[b * 4 + 3] != 0;
    s->finished = all;
  }
  return CORA_OK;
}

extern "C" int cora_generate(cora_model* m, const int32_t* prompt, int32_t B, int32_t P, int32_t gen_len,
                             int32_t block_len, int32_t steps_per_block, float tau, int32_t K, int32_t* tokens_out,
                             int64_t* passes_out, int64_t* batched_passes_out) {
  return cora_generate_ex(m, prompt, B, P, gen_len, block_len, steps_per_block, tau, K, nullptr, tokens_out,
                          passes_out, batched_passes_out);
}

extern "C" int cora_generate_ex(cora_model* m, const int32_t* prompt, int32_t B, int32_t P, int32_t gen_len,
                                int32_t block_len, int32_t steps_per_block, float tau, int32_t K,
                                const cora_decode_options* opt, int32_t* tokens_out, int64_t* passes_out,
                                int64_t* batched_passes_out) {
  REQUIRE(m && tokens_out && passes_out, "cora_generate: NULL argument");
  const cora_decode_options o = opt ? *opt : cora_decode_options{CORA_SCHEDULE_FIXED, CORA_PERSIST_BLOCK, -1, CORA_CACHE_NONE};
  cora_session* s = m->cached;
  // tau, K and the options are baked into the captured graphs, so they are part of the key.
  if (s && (s->B != B || s->P != P || s->G != gen_len || s->BL != block_len || s->T != steps_per_block ||
            s->tau != tau || s->K != K || s->opt.schedule != o.schedule || s->opt.persistence != o.persistence ||
            s->opt.eos_id != o.eos_id || s->opt.cache != o.cache)) {
    cora_session_destroy(s);
    s = nullptr;
  }
  int rc;
  if (!s) {
    rc = cora_session_create_ex(m, B, prompt, P, gen_len, block_len, steps_per_block, tau, K, &o, &s);
    if (rc) return rc;
    m->cached = s;
  } else {
    rc = cora_session_reset(s, prompt);
    if (rc) return rc;
  }
  rc = cora_session_run(s, nullptr, nullptr);
  if (rc) return rc;
  CK(cudaMemcpy2D(tokens_out, size_t(gen_len) * 4, s->tokens + P, size_t(s->S) * 4, size_t(gen_len) * 4, B,
                  cudaMemcpyDeviceToHost));
  std::vector<int32_t> ctrl(size_t(B) * 4);
  CK(cudaMemcpy(ctrl.data(), s->ctrl, ctrl.size() * 4, cudaMemcpyDeviceToHost));
  for (int b = 0; b < B; ++b) passes_out[b] = ctrl[size_t(b) * 4 + 2];
  if (batched_passes_out) *batched_passes_out = s->batched_passes;
  return CORA_OK;
}

// ---------------------------------------------------------- standalone ops
extern "C" int cora_gate_transfer(const float* conf, const int32_t* argmax, int32_t* prev, int32_t* persist,
                                  uint8_t* state, int32_t* tokens, int32_t B, int32_t R, int32_t k, float tau,
                                  int32_t K, uint8_t* unmask, uint8_t* accept, uint8_t* done, void* stream) {
  REQUIRE(conf && argmax && prev && persist && state && tokens && unmask && accept && done,
          "cora_gate_transfer: NULL pointer");
  REQUIRE(B >= 1 && R >= 1 && R <= 32, "cora_gate_transfer: need B >= 1 and 1 <= R <= 32");
  REQUIRE(k >= 0, "cora_gate_transfer: k must be >= 0");
  GateBuffers gb{const_cast<float*>(conf), const_cast<int32_t*>(argmax), prev, persist, state, tokens, unmask, accept,
                 done};
  launch_gate_transfer(gb, B, R, k, tau, K, static_cast<cudaStream_t>(stream));
  CK(cudaGetLastError());
  return CORA_OK;
}

extern "C" int cora_reduce_top1(const uint16_t* logits, int32_t rows, int32_t V, float* conf, int32_t* argmax,
                                void* stream) {
  REQUIRE(logits && conf && argmax, "cora_reduce_top1: NULL pointer");
  REQUIRE(rows >= 1 && V >= 1, "cora_reduce_top1: rows and V must be >= 1");
  REQUIRE(V % 8 != 0 || aligned16(logits), "cora_reduce_top1: logits must be 16-byte aligned");
  DeviceCtx* dc = nullptr;
  int rc = device_ctx(&dc);
  if (rc) return rc;
  const int n = reduce_top1_parts_count(rows, V, dc->num_sms);
  Top1Part* parts = nullptr;
  int* counters = nullptr;
  rc = reduce_scratch(dc, n, rows, rows, &parts, &counters);
  if (rc) return rc;
  GateBuffers gb{conf, argmax, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr};
  launch_reduce_fused(logits, rows, V, n, parts, counters, gb, 1, 0, 0.f, 0, false, static_cast<cudaStream_t>(stream));
  CK(cudaGetLastError());
  return CORA_OK;
}

extern "C" int cora_reduce_gate(const uint16_t* logits, int32_t B, int32_t R, int32_t V, float* conf, int32_t* argmax,
                                int32_t* prev, int32_t* persist, uint8_t* state, int32_t* tokens, int32_t k, float tau,
                                int32_t K, uint8_t* unmask, uint8_t* accept, uint8_t* done, void* stream) {
  REQUIRE(logits && conf && argmax && prev && persist && state && tokens && unmask && accept && done,
          "cora_reduce_gate: NULL pointer");
  REQUIRE(B >= 1 && R >= 1 && R <= 32 && V >= 1 && k >= 0, "cora_reduce_gate: bad shape");
  REQUIRE(V % 8 != 0 || aligned16(logits), "cora_reduce_gate: logits must be 16-byte aligned");
  DeviceCtx* dc = nullptr;
  int rc = device_ctx(&dc);
  if (rc) return rc;
  const int rows = B * R;
  const int n = reduce_top1_parts_count(rows, V, dc->num_sms);
  Top1Part* parts = nullptr;
  int* counters = nullptr;
  rc = reduce_scratch(dc, n, rows, B, &parts, &counters);
  if (rc) return rc;
  GateBuffers gb{conf, argmax, prev, persist, state, tokens, unmask, accept, done};
  launch_reduce_fused(logits, rows, V, n, parts, counters, gb, R, k, tau, K, true, static_cast<cudaStream_t>(stream));
  CK(cudaGetLastError());
  return CORA_OK;
}

extern "C" int cora_gemm_plan(int32_t M, int32_t N, int32_t K, int32_t epilogue, int32_t num_sms, int32_t* info,
                              int32_t* seg, int32_t cap, int32_t* n_seg) {
  REQUIRE(info && n_seg && (seg || cap == 0), "cora_gemm_plan: NULL pointer");
  REQUIRE(M >= 1 && num_sms >= 2 && K >= 64 && K % 64 == 0 && N >= 128 && N % 128 == 0 && cap >= 0,
          "cora_gemm_plan: bad M/N/K/num_sms/cap");
  REQUIRE(epilogue >= 0 && epilogue <= 3, "cora_gemm_plan: bad epilogue");
  REQUIRE(epilogue != CORA_EPI_SWIGLU || N % 256 == 0, "cora_gemm_plan: SWIGLU needs N %% 256 == 0");
  *n_seg = gemm_plan(M, N, K, epilogue, num_sms, info, seg, cap);
  return CORA_OK;
}

extern "C" int cora_op_gemm(const uint16_t* A, const uint16_t* B, void* C, int32_t M, int32_t N, int32_t K,
                            int32_t ldc, int32_t epilogue, const float* rope, int32_t seq, int32_t head_dim,
                            int32_t rope_cols, void* stream) {
  REQUIRE(A && B && C, "cora_op_gemm: NULL pointer");
  REQUIRE(M >= 1 && N >= 128 && N % 128 == 0 && K >= 64 && K % 64 == 0, "cora_op_gemm: bad M/N/K");
  REQUIRE(epilogue >= 0 && epilogue <= 3, "cora_op_gemm: bad epilogue");
  REQUIRE(epilogue != CORA_EPI_SWIGLU || N % 256 == 0, "cora_op_gemm: SWIGLU needs N %% 256 == 0");
  REQUIRE(aligned16(A) && aligned16(B) && aligned16(C), "cora_op_gemm: pointers must be 16-byte aligned");
  const int out_cols = epilogue == CORA_EPI_SWIGLU ? N / 2 : N;
  REQUIRE(ldc >= out_cols && ldc % 8 == 0, "cora_op_gemm: bad ldc");
  if (epilogue == CORA_EPI_ROPE_BF16) {
    REQUIRE(rope && seq >= 1 && (head_dim == 64 || head_dim == 128) && gemm_block_n(N, epilogue) % head_dim == 0,
            "cora_op_gemm: bad RoPE arguments");
  }
  DeviceCtx* dc = nullptr;
  int rc = device_ctx(&dc);
  if (rc) return rc;
  if ((rc = kernels_prepare())) return rc;
  CUtensorMap ta, tb, tc;
  if (!make_tmap_bf16_2d(&ta, A, M, K, size_t(K) * 2, 128, 64) || !make_tmap_bf16_2d(&tb, B, N, K, size_t(K) * 2, 128, 64) ||
      !make_gemm_out_tmap(&tc, C, M, ldc, epilogue))
    return fail(CORA_ECUDA, "cora_op_gemm: tensor map encoding failed");
  GemmEpilogue ep{C, ldc, epilogue, rope, seq, head_dim, rope_cols, 0};
  ep.a_ptr = A;
  ep.a_rows = M;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  float* rope_t = nullptr;
  if (epilogue == CORA_EPI_ROPE_BF16) {
    // the row-tiled epilogue reads the table frequency-major: a stream-ordered
    // transposed copy, released after the GEMM
    CK(cudaMallocAsync(reinterpret_cast<void**>(&rope_t), size_t(seq) * head_dim * sizeof(float), st));
    launch_rope_transpose(rope, rope_t, seq, head_dim / 2, st);
    ep.rope_t = rope_t;
    ep.rope_tn = seq;
  }
  const cudaError_t ge = launch_gemm(ta, tb, tc, M, N, K, ep, dc->gemm_ws, dc->err, dc->num_sms, st);
  if (rope_t) CK(cudaFreeAsync(rope_t, st));
  CK(ge);
  return CORA_OK;
}

extern "C" int cora_op_attention_rows(const uint16_t* qkv, uint16_t* out, int32_t B, int32_t S, int32_t Hq,
                                      int32_t Hkv, int32_t hd, int32_t q_start, int32_t q_len, void* stream);

extern "C" int cora_op_attention(const uint16_t* qkv, uint16_t* out, int32_t B, int32_t S, int32_t Hq, int32_t Hkv,
                                 int32_t hd, void* stream) {
  return cora_op_attention_rows(qkv, out, B, S, Hq, Hkv, hd, 0, S, stream);
}

extern "C" int cora_op_attention_rows(const uint16_t* qkv, uint16_t* out, int32_t B, int32_t S, int32_t Hq,
                                      int32_t Hkv, int32_t hd, int32_t q_start, int32_t q_len, void* stream) {
  REQUIRE(qkv && out, "cora_op_attention: NULL pointer");
  REQUIRE(B >= 1 && S >= 1 && Hq >= 1 && Hkv >= 1 && Hq % Hkv == 0 && (hd == 64 || hd == 128),
          "cora_op_attention: bad shape");
  REQUIRE(q_start >= 0 && q_len >= 1 && int64_t(q_start) + q_len <= S, "cora_op_attention: bad query range");
  REQUIRE(aligned16(qkv) && aligned16(out), "cora_op_attention: pointers must be 16-byte aligned");
  int rc = kernels_prepare();
  if (rc) return rc;
  DeviceCtx* dc = nullptr;
  if ((rc = device_ctx(&dc))) return rc;
  CUtensorMap tq;
  const size_t cols = size_t(Hq + 2 * Hkv) * hd;
  if (!make_tmap_bf16_2d(&tq, qkv, size_t(B) * S, cols, cols * 2, 128, 64))
    return fail(CORA_ECUDA, "cora_op_attention: tensor map encoding failed");
  CK(launch_attention_tc(tq, out, B, S, Hq, Hkv, hd, q_start, q_len, dc->err, dc->num_sms,
                         static_cast<cudaStream_t>(stream)));
  CK(cudaGetLastError());
  return CORA_OK;
}

extern "C" int cora_op_rmsnorm(const float* x, const uint16_t* w, uint16_t* out, int32_t M, int32_t d, float eps,
                               void* stream) {
  REQUIRE(x && out, "cora_op_rmsnorm: NULL pointer");
  REQUIRE(M >= 1 && d >= 8 && d % 8 == 0, "cora_op_rmsnorm: bad shape");
  REQUIRE(aligned16(x) && aligned16(out) && (!w || aligned16(w)), "cora_op_rmsnorm: pointers must be 16-byte aligned");
  launch_rmsnorm(x, w, out, M, d, eps, static_cast<cudaStream_t>(stream));
  CK(cudaGetLastError());
  return CORA_OK;
}

extern "C" int cora_op_lm_head_top1(const uint16_t* x, const uint16_t* W, int32_t R, int32_t V, int32_t d, float* conf,
                                    int32_t* argmax, void* stream) {
  REQUIRE(x && W && conf && argmax, "cora_op_lm_head_top1: NULL pointer");
  REQUIRE(R >= 1 && R <= 256 && V >= 1 && d >= 64 && d % 64 == 0, "cora_op_lm_head_top1: bad shape");
  REQUIRE(aligned16(x) && aligned16(W), "cora_op_lm_head_top1: pointers must be 16-byte aligned");
  DeviceCtx* dc = nullptr;
  int rc = device_ctx(&dc);
  if (rc) return rc;
  if ((rc = kernels_prepare())) return rc;
  CUtensorMap tw, tx;
  if (!make_tmap_bf16_2d(&tw, W, V, d, size_t(d) * 2, 128, 64) ||
      !make_tmap_bf16_2d(&tx, x, R, d, size_t(d) * 2, lm_head_npad(R), 64))
    return fail(CORA_ECUDA, "cora_op_lm_head_top1: tensor map encoding failed");
  const int n = lm_head_parts_count(V, dc->num_sms);
  void* parts = nullptr;
  rc = scratch_reserve(dc, size_t(n) * R * sizeof(Top1Part), &parts);
  if (rc) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  CK(launch_lm_head_top1(tw, tx, R, V, d, static_cast<Top1Part*>(parts), n, dc->err, st));
  launch_combine_top1(static_cast<Top1Part*>(parts), n, R, conf, argmax, st);
  CK(cudaGetLastError());
  return CORA_OK;
}

extern "C" int cora_synth_normal_bf16(uint16_t* out, int64_t count, uint64_t key, int64_t start, float scale,
                                      void* stream) {
  REQUIRE(out && count >= 0 && start >= 0, "cora_synth_normal_bf16: bad argument");
  launch_synth_normal_bf16(out, count, key, start, scale, static_cast<cudaStream_t>(stream));
  CK(cudaGetLastError());
  return CORA_OK;
}

extern "C" int cora_check_wait_timeout(int32_t which, int32_t* code_out) {
  REQUIRE(code_out && (which == 0 || which == 1), "cora_check_wait_timeout: bad argument");
  DeviceCtx* dc = nullptr;
  int rc = device_ctx(&dc);
  if (rc) return rc;
  int* buf = nullptr;  // [0] the flag nothing sets, [1] this check's own error word
  CK(cudaMalloc(&buf, 2 * sizeof(int)));
  cudaError_t e = cudaMemset(buf, 0, 2 * sizeof(int));
  if (e == cudaSuccess) e = launch_wait_check(which, buf, buf + 1, 0);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  int code = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&code, buf + 1, sizeof(int), cudaMemcpyDeviceToHost);
  cudaFree(buf);
  CK(e);
  *code_out = code;
  return CORA_OK;
}

extern "C" int cora_device_error(int32_t* code, int32_t clear) {
  REQUIRE(code, "cora_device_error: NULL pointer");
  DeviceCtx* dc = nullptr;
  int rc = device_ctx(&dc);
  if (rc) return rc;
  CK(cudaDeviceSynchronize());
  CK(cudaMemcpy(code, dc->err, sizeof(int), cudaMemcpyDeviceToHost));
  if (clear) CK(cudaMemset(dc->err, 0, sizeof(int)));
  return CORA_OK;
}
