// Seeded weight fill, token embedding and RMSNorm kernels.
#include "cora_device.cuh"
#include "cora_kernels.h"

namespace cora {

// SplitMix64 output function (Steele, Lea and Flood, OOPSLA 2014).
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

// Element i = bf16(fp32(X) * scale), X = 2 * (sum of the four 16-bit fields of
// output start+i of stream `key`) - 4 * 65535; rounding to nearest even.
__global__ void synth_normal_bf16_kernel(uint16_t* __restrict__ out, int64_t count, uint64_t key, int64_t start,
                                         float scale) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < count; i += stride) {
    const uint64_t z = mix64(key + static_cast<uint64_t>(start + i + 1) * 0x9E3779B97F4A7C15ULL);
    const uint32_t s = static_cast<uint32_t>(z & 0xFFFF) + static_cast<uint32_t>((z >> 16) & 0xFFFF) +
                       static_cast<uint32_t>((z >> 32) & 0xFFFF) + static_cast<uint32_t>(z >> 48);
    const int32_t x = 2 * static_cast<int32_t>(s) - 4 * 65535;
    uint32_t u = __float_as_uint(__fmul_rn(static_cast<float>(x), scale));
    u += 0x7FFFu + ((u >> 16) & 1u);
    out[i] = static_cast<uint16_t>(u >> 16);
  }
}

// dst[r, c] = bf16(src[r, c]) for a [rows, cols] fp32 block (row strides in
// elements), round to nearest even: the fp32 weight input of the model.
__global__ void f32_to_bf16_2d_kernel(const float* __restrict__ src, int64_t src_ld, uint16_t* __restrict__ dst,
                                      int64_t dst_ld, int64_t rows, int64_t cols) {
  const int64_t n = rows * cols;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += stride) {
    const int64_t r = i / cols, c = i - r * cols;
    dst[r * dst_ld + c] = __bfloat16_as_ushort(__float2bfloat16_rn(src[r * src_ld + c]));
  }
}

// h[r, :] = float(embed[tokens[r], :]); one warp per row, 16-byte loads.
// Row r of h takes token r of the canvas, or, with rows_per_seq > 0 (packed
// rows of a prefix-cache pass), token lo + r % rows_per_seq of sequence
// r / rows_per_seq (canvas rows S_tok apart).
__global__ void embed_kernel(const int32_t* __restrict__ tokens, const uint16_t* __restrict__ embed,
                             float* __restrict__ h, int M, int d, int S_tok, int lo, int rows_per_seq) {
  pdl_trigger();
  pdl_wait();
  const int row = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  const int64_t ti = rows_per_seq > 0
                         ? static_cast<int64_t>(row / rows_per_seq) * S_tok + lo + row % rows_per_seq
                         : static_cast<int64_t>(row);
  const int tok = tokens[ti];
  const uint4* src = reinterpret_cast<const uint4*>(embed + static_cast<int64_t>(tok) * d);
  float4* dst = reinterpret_cast<float4*>(h + static_cast<int64_t>(row) * d);
  for (int c = lane; c < d / 8; c += 32) {
    const uint4 v = src[c];
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    float f[8];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      f[2 * j] = __uint_as_float(w[j] << 16);
      f[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
    }
    dst[2 * c] = make_float4(f[0], f[1], f[2], f[3]);
    dst[2 * c + 1] = make_float4(f[4], f[5], f[6], f[7]);
  }
}

// One warp normalises one fp32 row of length d (d % 8 == 0) into bf16.
__device__ __forceinline__ void rmsnorm_row_warp(const float* __restrict__ x, const uint16_t* __restrict__ w,
                                                 uint16_t* __restrict__ out, int d, float eps, int lane) {
  const float4* xv = reinterpret_cast<const float4*>(x);
  float ss = 0.f;
  for (int c = lane; c < d / 4; c += 32) {
    const float4 v = xv[c];
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float r = rsqrtf(ss / static_cast<float>(d) + eps);
  uint2* ov = reinterpret_cast<uint2*>(out);
  for (int c = lane; c < d / 4; c += 32) {
    const float4 v = xv[c];
    float g0 = 1.f, g1 = 1.f, g2 = 1.f, g3 = 1.f;
    if (w) {
      const uint2 wv = reinterpret_cast<const uint2*>(w)[c];
      g0 = __uint_as_float(wv.x << 16);
      g1 = __uint_as_float(wv.x & 0xFFFF0000u);
      g2 = __uint_as_float(wv.y << 16);
      g3 = __uint_as_float(wv.y & 0xFFFF0000u);
    }
    ov[c] = make_uint2(pack_bf16x2(v.x * r * g0, v.y * r * g1), pack_bf16x2(v.z * r * g2, v.w * r * g3));
  }
}

// One 128-thread CTA per row (d <= 4096, d % 4 == 0): the row is read once
// into registers (up to 8 float4 per thread), reduced, scaled, stored.
constexpr int kNormThreads = 128;
constexpr int kNormVec = 8;

__device__ __forceinline__ void rmsnorm_row_cta(const float* __restrict__ x, const uint16_t* __restrict__ w,
                                                uint16_t* __restrict__ out, int d, float eps) {
  const float4* xv = reinterpret_cast<const float4*>(x);
  const int nv = d >> 2;
  float4 v[kNormVec];
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < kNormVec; ++i) {
    const int c = threadIdx.x + i * kNormThreads;
    v[i] = c < nv ? xv[c] : make_float4(0.f, 0.f, 0.f, 0.f);
    ss += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  __shared__ float part[kNormThreads / 32];
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int i = 0; i < kNormThreads / 32; ++i) tot += part[i];
  const float r = rsqrtf(tot / static_cast<float>(d) + eps);
  uint2* ov = reinterpret_cast<uint2*>(out);
#pragma unroll
  for (int i = 0; i < kNormVec; ++i) {
    const int c = threadIdx.x + i * kNormThreads;
    if (c < nv) {
      float g0 = 1.f, g1 = 1.f, g2 = 1.f, g3 = 1.f;
      if (w) {
        const uint2 wv = reinterpret_cast<const uint2*>(w)[c];
        g0 = __uint_as_float(wv.x << 16);
        g1 = __uint_as_float(wv.x & 0xFFFF0000u);
        g2 = __uint_as_float(wv.y << 16);
        g3 = __uint_as_float(wv.y & 0xFFFF0000u);
      }
      ov[c] = make_uint2(pack_bf16x2(v[i].x * r * g0, v[i].y * r * g1), pack_bf16x2(v[i].z * r * g2, v[i].w * r * g3));
    }
  }
}

__global__ void __launch_bounds__(kNormThreads) rmsnorm_kernel(const float* __restrict__ x,
                                                                const uint16_t* __restrict__ w,
                                                                uint16_t* __restrict__ out, int M, int d, float eps) {
  pdl_trigger();
  pdl_wait();
  const int row = blockIdx.x;
  if (d <= 4 * kNormThreads * kNormVec) {
    rmsnorm_row_cta(x + static_cast<int64_t>(row) * d, w, out + static_cast<int64_t>(row) * d, d, eps);
  } else if (threadIdx.x < 32) {  // wider rows: one warp, two passes
    rmsnorm_row_warp(x + static_cast<int64_t>(row) * d, w, out + static_cast<int64_t>(row) * d, d, eps,
                     threadIdx.x & 31);
  }
}

// Final RMSNorm on the active block's rows only: row i of sequence b is canvas
// position prompt_len + block(b) * block_len + i.  Finished sequences keep
// their last block (their rows are computed and ignored).
// Final RMSNorm of the rows Eq. 1 needs: rows_per_seq == BL takes each
// sequence's active block; otherwise (rows_per_seq == G) every generation
// position, for the carry-over persistence variant.
__global__ void final_norm_rows_kernel(const float* __restrict__ h, const uint16_t* __restrict__ w,
                                       const int32_t* __restrict__ ctrl, uint16_t* __restrict__ out, int B, int S,
                                       int P, int BL, int n_blocks, int d, float eps, int rows_per_seq) {
  // P < 0: h holds packed prefix-cache rows, S per sequence, with the active
  // block first.
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  if (r >= B * rows_per_seq) return;
  const int b = r / rows_per_seq, i = r % rows_per_seq;
  int64_t src = static_cast<int64_t>(b) * S + (P < 0 ? 0 : P) + i;
  if (rows_per_seq == BL && P >= 0) {
    int blk = ctrl[b * 4 + 0];
    blk = blk < n_blocks ? blk : n_blocks - 1;
    src += static_cast<int64_t>(blk) * BL;
  }
  rmsnorm_row_warp(h + src * d, w, out + static_cast<int64_t>(r) * d, d, eps, threadIdx.x & 31);
}

// Canvas = [prompt | mask_id ...] per sequence; every position unresolved,
// fresh persistence state, block/step/pass counters zero.
__global__ void session_init_kernel(int32_t* __restrict__ tokens, const int32_t* __restrict__ prompt,
                                    uint8_t* __restrict__ state, int32_t* __restrict__ persist,
                                    int32_t* __restrict__ prev, int32_t* __restrict__ ctrl,
                                    int32_t* __restrict__ status, int B, int P, int S, int G, int BL, int mask_id) {
  const int64_t n = static_cast<int64_t>(B) * S;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int b = static_cast<int>(i / S), p = static_cast<int>(i % S);
    tokens[i] = p < P ? prompt[static_cast<int64_t>(b) * P + p] : mask_id;
    if (p >= P) state[static_cast<int64_t>(b) * G + (p - P)] = 0;
  }
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t < B * BL) {
    persist[t] = 0;
    prev[t] = -1;
  }
  if (t < B * 4) ctrl[t] = 0;
  if (t < 4) status[t] = t == 3 ? 1 : 0;  // {all_done, error word, loop counter, next pass: dense, block 0}
}

}  // namespace cora

using namespace cora;

void launch_session_init(int32_t* tokens, const int32_t* prompt, uint8_t* state, int32_t* persist, int32_t* prev,
                         int32_t* ctrl, int32_t* status, int B, int P, int S, int G, int BL, int mask_id,
                         cudaStream_t st) {
  const int64_t n = static_cast<int64_t>(B) * S;
  int64_t blocks = (n + 255) / 256;
  const int64_t need = (static_cast<int64_t>(B) * (BL > 4 ? BL : 4) + 255) / 256;
  if (blocks < need) blocks = need;
  if (blocks > 4096) blocks = 4096 > need ? 4096 : need;
  session_init_kernel<<<static_cast<int>(blocks), 256, 0, st>>>(tokens, prompt, state, persist, prev, ctrl, status, B,
                                                                 P, S, G, BL, mask_id);
}

void launch_f32_to_bf16_2d(const float* src, int64_t src_ld, uint16_t* dst, int64_t dst_ld, int64_t rows,
                           int64_t cols, cudaStream_t st) {
  const int64_t n = rows * cols;
  int64_t blocks = (n + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  f32_to_bf16_2d_kernel<<<static_cast<int>(blocks), 256, 0, st>>>(src, src_ld, dst, dst_ld, rows, cols);
}

void launch_synth_normal_bf16(uint16_t* out, int64_t count, uint64_t key, int64_t start, float scale,
                              cudaStream_t st) {
  if (count <= 0) return;
  int64_t blocks = (count + 255) / 256;
  if (blocks > 152 * 64) blocks = 152 * 64;
  synth_normal_bf16_kernel<<<static_cast<int>(blocks), 256, 0, st>>>(out, count, key, start, scale);
}

void launch_embed(const int32_t* tokens, const uint16_t* embed, float* h, int M, int d, int S_tok, int lo,
                  int rows_per_seq, cudaStream_t st) {
  launch_pdl(embed_kernel, dim3((M + 7) / 8), dim3(256), 0, st, tokens, embed, h, M, d, S_tok, lo, rows_per_seq);
}

void launch_rmsnorm(const float* x, const uint16_t* w, uint16_t* out, int M, int d, float eps, cudaStream_t st) {
  launch_pdl(rmsnorm_kernel, dim3(M), dim3(kNormThreads), 0, st, x, w, out, M, d, eps);
}

void launch_final_norm_rows(const float* h, const uint16_t* w, const int32_t* ctrl, uint16_t* out, int B, int S,
                            int P, int BL, int n_blocks, int d, float eps, int rows_per_seq, cudaStream_t st) {
  const int R = B * rows_per_seq;
  launch_pdl(final_norm_rows_kernel, dim3((R + 7) / 8), dim3(256), 0, st, h, w, ctrl, out, B, S, P, BL, n_blocks, d,
             eps, rows_per_seq);
}
