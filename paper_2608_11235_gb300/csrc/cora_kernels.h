// Internal host-side launchers shared by the library's translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace cora {
struct Top1;

// Launches `kernel` with programmatic stream serialization, so it may begin
// while its predecessor in the stream finishes (each kernel calls pdl_wait()
// before its first global-memory access).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
}

// Partial Eq. 1 state of one row over part of the vocabulary (see Top1 in
// cora_device.cuh): running max logit, sum of exp(logit - max), lowest index
// of the max.  Layout of a partial array: [n_parts][rows].
struct Top1Part {
  float m;
  float s;
  int32_t idx;
};

// Gate launch parameters for the session path (one warp per sequence).
struct SessionGateArgs {
  const Top1Part* parts;  // Eq. 1 partials, chunked (see rows_per_seq)
  int n_parts;
  int32_t* ctrl;          // [B][4] {block, step, passes, finished}
  int32_t* tokens;        // [B][S]
  uint8_t* state;         // [B][G]
  int32_t* persist;       // [B][rows_per_seq]
  int32_t* prev;          // [B][rows_per_seq]
  float* conf;            // [B][rows_per_seq]
  int32_t* argmax;        // [B][rows_per_seq]
  uint8_t* unmask;        // [B][BL]
  uint8_t* accept;        // [B][BL]
  uint8_t* all_done;      // [1]
  uint8_t* blk_done;      // [B]: 1 when the sequence's block has no unresolved position after the step
  int* err;
  int B, S, P, G, BL, T;
  float tau;
  int K;
  int schedule;  // CORA_SCHEDULE_*
  int eos_id;    // < 0: none
  // Eq. 1 rows: rows_per_seq per sequence (BL: the active block; G: every
  // generation position, carry-over persistence), their partials in chunks of
  // chunk_rows rows ([n_chunks][n_parts][chunk_rows], the last chunk shorter).
  int rows_per_seq;
  int chunk_rows;
  // Prefix-cache mode: sequences move to the next block together (a sequence
  // whose block has ended waits, ctrl step = -1); the kernel publishes the
  // next pass in status[3] (bit 0: a block's first, dense pass; bits 1..: block).
  int lockstep;
};

// dst (bf16 bits, row stride dst_ld elements) = round-to-nearest-even of the
// fp32 block src [rows, cols] (row stride src_ld elements); device pointers.
void launch_f32_to_bf16_2d(const float* src, int64_t src_ld, uint16_t* dst, int64_t dst_ld, int64_t rows,
                           int64_t cols, cudaStream_t st);
void launch_synth_normal_bf16(uint16_t* out, int64_t count, uint64_t key, int64_t start, float scale,
                              cudaStream_t st);
void launch_embed(const int32_t* tokens, const uint16_t* embed, float* h, int M, int d, int S_tok, int lo,
                  int rows_per_seq, cudaStream_t st);
void launch_rmsnorm(const float* x, const uint16_t* w, uint16_t* out, int M, int d, float eps, cudaStream_t st);
void launch_final_norm_rows(const float* h, const uint16_t* w, const int32_t* ctrl, uint16_t* out, int B, int S,
                            int P, int BL, int n_blocks, int d, float eps, int rows_per_seq, cudaStream_t st);

// Gate buffers of B blocks of R positions ([B, R] each; done is [B]).
struct GateBuffers {
  float* conf;
  int32_t* argmax;
  int32_t* prev;
  int32_t* persist;
  uint8_t* state;
  int32_t* tokens;
  uint8_t* unmask;
  uint8_t* accept;
  uint8_t* done;
};

// Eq. 1 from materialised bf16 logits [rows, V], grid (n_chunks, rows), with
// the combine (and, when gate is set, the transfer rule + Eq. 2-4 of each
// block of R rows) done by the last CTA of each group.  counters: zeroed ints,
// one per row (gate == false) or per block (gate == true); left zeroed.
int reduce_top1_parts_count(int rows, int V, int num_sms);
int cora_set_error(int code, const char* msg);
void launch_reduce_fused(const uint16_t* logits, int rows, int V, int n_chunks, Top1Part* parts, int* counters,
                         const GateBuffers& gb, int R, int k, float tau, int K, bool gate, cudaStream_t st);
void launch_combine_top1(const Top1Part* parts, int n_parts, int rows, float* conf, int32_t* argmax,
                         cudaStream_t st);
void launch_gate_transfer(const GateBuffers& gb, int B, int R, int k, float tau, int K, cudaStream_t st);
void launch_session_gate(const SessionGateArgs& a, cudaStream_t st);

// GEMM (tcgen05).  Epilogue parameters.
// rope [seq][half][2] -> rope_t [half][seq][2].
void launch_rope_transpose(const float* rope, float* rope_t, int seq, int half, cudaStream_t st);
struct GemmEpilogue {
  void* C;
  int ldc;
  int mode;             // CORA_EPI_*
  const float* rope;    // [seq][head_dim/2][2] (position-major; the few-row kernel)
  int seq;
  int head_dim;
  int rope_cols;
  // 1 when B is not written by any kernel that may still run on the stream
  // (model weights): the 2-CTA kernel then starts loading B before waiting
  // for the previous kernel (programmatic dependent launch).
  int b_static;
  // Set by launch_gemm: equal k-splits per tile (0 = stream-K) and their
  // skew toward the finishing piece, in k-blocks.
  int splits;
  int split_skew;
  int split_pair;  // 1: two k-pieces per tile, each finalising half of the columns
  // Set by launch_gemm: whole tiles per unit (CTA pair) run in data-parallel
  // waves after the stream-K tiles, the row blocks per group of the tile
  // numbering (1: M-slowest), and the units sharing the stream-K tiles.
  int dp_waves;
  int raster_group;
  int sk_units;
  // ROPE epilogue on packed prefix-cache rows: row r is position
  // rope_pos0 + r % seq of sequence r / seq; with out3d, C is a 3-D map
  // [sequence][position][column] and row r is stored at that position.
  int rope_pos0;
  int out3d;
  // A (row-major [a_rows, K] bf16): with it, launch_gemm routes M <= 64 to
  // the few-row (swap-AB) kernel; out_rows_per_seq = output rows per
  // sequence for out3d stores there.
  const void* a_ptr;
  int64_t a_rows;
  int out_rows_per_seq;
  // The same RoPE table frequency-major, [head_dim/2][rope_tn][2]: the
  // row-tiled kernels' epilogue thread owns one row (position), so a warp
  // reads one frequency for 32 consecutive positions in one 256-byte line
  // pair instead of 32 lines.
  const float* rope_t;
  int rope_tn;
};

// Stream-K workspace: one fp32 partial slot of 128 x 256 per CTA plus one
// flag per CTA (zero between launches).
struct GemmWorkspace {
  float* partial;
  int* flags;
};
size_t gemm_workspace_bytes(int num_sms);

// Tensor-map encoder (driver entry point fetched at runtime).
// Disagreement counts of a canvas against a reference canvas: out [B][3].
void launch_disagreement(const int32_t* tok, const uint8_t* state, const int32_t* ref, int B, int S, int P, int G,
                         long long* out, cudaStream_t st);

// One-thread kernel that sets the WHILE condition of the whole-decode graph.
cudaError_t launch_step_loop_cond(cudaGraphConditionalHandle h, int32_t* status, int32_t max_iters, cudaStream_t st);

bool make_tmap_bf16_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t row_stride_bytes,
                       uint32_t box_rows, uint32_t box_cols);
// 3-D bf16 map (innermost d0), 128-byte swizzle; strides of dims 1 and 2 in bytes.
bool make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t stride1_bytes,
                       uint64_t stride2_bytes, uint32_t b0, uint32_t b1, uint32_t b2);

int gemm_block_n(int N, int mode);
// Failure-detection self-check (see cora_check_wait_timeout).
cudaError_t launch_wait_check(int which, const int* flag, int* err, cudaStream_t st);
// Host-side plan of launch_gemm's work split (see cora_gemm_plan); returns the
// number of segments, writes info[7] and up to cap segments of 6 ints.
int gemm_plan(int M, int N, int K, int mode, int num_sms, int* info, int* seg, int cap);
cudaError_t launch_gemm(const CUtensorMap& tmA, const CUtensorMap& tmB, const CUtensorMap& tmC, int M, int N, int K,
                        const GemmEpilogue& ep, const GemmWorkspace& ws, int* err, int num_sms, cudaStream_t st);
bool make_gemm_out_tmap(CUtensorMap* map, void* C, int M, int ldc, int mode);
// Few-row GEMM (gemm_skinny.cu): tmW = weights [N, K] (boxes of 128 rows x 64),
// tmX = A with boxes of gemm_skinny_npad(M) rows x 64.
int gemm_skinny_npad(int M);
bool gemm_skinny_supported(int M, int N, int K, const GemmEpilogue& ep);
cudaError_t launch_gemm_skinny(const CUtensorMap& tmW, const CUtensorMap& tmX, int M, int N, int K,
                               const GemmEpilogue& ep, const GemmWorkspace& ws, int* err, int num_sms,
                               cudaStream_t st);
// GemmWorkspace.flags entries: the row-tiled kernels' flags, then the
// few-row kernel's tile tickets.
constexpr int kGemmFlagCount = 1024;
// Generic 2-D tensor map (element size 2 = bf16, 4 = fp32), 128-byte swizzle.
bool make_tmap_2d(CUtensorMap* map, const void* base, int elem_bytes, uint64_t rows, uint64_t cols,
                  uint64_t row_stride_bytes, uint32_t box_rows, uint32_t box_cols);

// Fused LM head + Eq. 1 partials: x [R, d] (tensor map box rows = n_pad),
// W [V, d].  Writes parts [grid][R]; returns the number of parts used.
int lm_head_parts_count(int V, int num_sms);
int lm_head_npad(int R);
cudaError_t launch_lm_head_top1(const CUtensorMap& tmW, const CUtensorMap& tmX, int R, int V, int d,
                                Top1Part* parts, int n_parts, int* err, cudaStream_t st);

// Shared-memory attributes of the big-smem kernels (call once per device,
// outside stream capture).
cudaError_t gemm_prepare();
cudaError_t lm_head_prepare();
cudaError_t attention_tc_prepare();
cudaError_t attention_tc2_prepare();
// Two query tiles per CTA, persistent over (sequence, head, query-tile pair)
// items; out bf16 [B][q_len][Hq*128] written directly.
cudaError_t launch_attention_tc2(const CUtensorMap& tmQKV, uint16_t* out, int B, int S, int Hq, int Hkv, int q_start,
                                 int q_len, int* err, int num_sms, cudaStream_t st);
// tcgen05 attention, head_dim hd in {64, 128}; tmQKV: bf16 [B*S, (Hq+2Hkv)*hd], box 128 rows x 64 cols.
// Queries q_start .. q_start + q_len - 1 of every sequence against all S keys;
// out holds q_len rows per sequence ((0, S): the dense pass).  Items =
// ceil(q_len/128) * Hq * B: one CTA per item (hd 64; hd 128 when they fit on
// the SMs), else the two-query-tile persistent kernel (launch_attention_tc2).
cudaError_t launch_attention_tc(const CUtensorMap& tmQKV, uint16_t* out, int B, int S, int Hq, int Hkv, int hd,
                                int q_start, int q_len, int* err, int num_sms, cudaStream_t st);

void launch_session_init(int32_t* tokens, const int32_t* prompt, uint8_t* state, int32_t* persist, int32_t* prev,
                         int32_t* ctrl, int32_t* status, int B, int P, int S, int G, int BL, int mask_id,
                         cudaStream_t st);


