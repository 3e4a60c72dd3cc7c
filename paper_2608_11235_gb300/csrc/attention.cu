// Bidirectional (non-causal) softmax attention, flash-style: every query of a
// sequence attends to every key of that sequence; K/V tiles stream through
// shared memory (cp.async, double-buffered, XOR-swizzled 16-byte chunks) and
// the softmax is computed online in registers (running max and sum).
// Grid: (ceil(S/64) query tiles, Hq, B); 4 warps x 16 query rows.
// Query head h reads KV head h / (Hq/Hkv) (grouped-query attention).
#include <math.h>

#include "cora_device.cuh"
#include "cora_kernels.h"

namespace cora {

constexpr int kQT = 64;   // query rows per CTA
constexpr int kKT = 64;   // keys per tile

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool pred) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(pred ? 16 : 0) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Byte offset of 16-byte chunk `ch` of row `r` in a [rows][HD] bf16 tile.
template <int HD>
__device__ __forceinline__ uint32_t swz(int r, int ch) {
  return static_cast<uint32_t>(r * (HD * 2) + ((ch ^ (r & 7)) << 4));
}

// Issue cp.async for a [64][HD] tile from rows row0.. of a strided bf16 matrix
// (rows beyond `nrows` are zero-filled).
template <int HD>
__device__ __forceinline__ void load_tile(uint32_t sbase, const uint16_t* g, int64_t ld, int row0, int nrows) {
  constexpr int CH = HD / 8;  // 16-byte chunks per row
  for (int i = threadIdx.x; i < 64 * CH; i += blockDim.x) {
    const int r = i / CH, ch = i % CH;
    const bool ok = row0 + r < nrows;
    const uint16_t* src = g + static_cast<int64_t>(ok ? row0 + r : 0) * ld + ch * 8;
    cp_async16(sbase + swz<HD>(r, ch), src, ok);
  }
}

template <int HD>
// Queries q_start .. q_start + q_len - 1 of each sequence (all S keys); the
// output row of query q is (q - q_start) of the sequence's q_len rows.
__global__ void __launch_bounds__(128) attention_kernel(const uint16_t* __restrict__ qkv, uint16_t* __restrict__ out,
                                                        int S, int Hq, int Hkv, int q_start, int q_len) {
  extern __shared__ __align__(128) uint16_t att_smem[];
  uint16_t* sQ = att_smem;                   // [64][HD]
  uint16_t* sK0 = sQ + kQT * HD;             // 2 x [64][HD]
  uint16_t* sV0 = sK0 + 2 * kKT * HD;        // 2 x [64][HD]

  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int kvh = h / (Hq / Hkv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t ld = static_cast<int64_t>(Hq + 2 * Hkv) * HD;
  const uint16_t* base = qkv + static_cast<int64_t>(b) * S * ld;
  const uint16_t* gQ = base + static_cast<int64_t>(h) * HD;
  const uint16_t* gK = base + static_cast<int64_t>(Hq + kvh) * HD;
  const uint16_t* gV = base + static_cast<int64_t>(Hq + Hkv + kvh) * HD;
  const int q0 = q_start + qt * kQT;
  const int q_end = q_start + q_len;
  const int n_kt = (S + kKT - 1) / kKT;

  pdl_trigger();
  pdl_wait();
  const uint32_t sq = smem_u32(sQ);
  const uint32_t sk[2] = {smem_u32(sK0), smem_u32(sK0 + kKT * HD)};
  const uint32_t sv[2] = {smem_u32(sV0), smem_u32(sV0 + kKT * HD)};

  load_tile<HD>(sq, gQ, ld, q0, S);
  load_tile<HD>(sk[0], gK, ld, 0, S);
  load_tile<HD>(sv[0], gV, ld, 0, S);
  cp_async_commit();
  cp_async_wait<0>();
  __syncthreads();

  // Q fragments of this warp's 16 rows (A operand, row-major).
  uint32_t qf[HD / 16][4];
  {
    const int r = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      const int ch = kk * 2 + (lane >> 4);
      ldsm_x4(sq + swz<HD>(r, ch), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
    }
  }

  const float sl2 = 1.4426950408889634f / sqrtf(static_cast<float>(HD));  // log2(e) / sqrt(hd)
  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;  // rows g and g+8

  for (int j = 0; j < n_kt; ++j) {
    const int buf = j & 1;
    if (j + 1 < n_kt) {
      load_tile<HD>(sk[buf ^ 1], gK, ld, (j + 1) * kKT, S);
      load_tile<HD>(sv[buf ^ 1], gV, ld, (j + 1) * kKT, S);
    }
    cp_async_commit();

    // S = Q K^T for 16 rows x 64 keys.
    float s[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        const int key = np * 16 + (lane & 7) + (lane >> 4) * 8;
        const int ch = kk * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(sk[buf] + swz<HD>(key, ch), b0, b1, b2, b3);
        mma_bf16_16816(s[2 * np], qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], b0, b1);
        mma_bf16_16816(s[2 * np + 1], qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], b2, b3);
      }
    }
    // Keys past the end of the sequence do not exist.
    const int kbase = j * kKT;
    if (kbase + kKT > S) {
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        const int key = kbase + n * 8 + (lane & 3) * 2;
        if (key >= S) s[n][0] = s[n][2] = -INFINITY;
        if (key + 1 >= S) s[n][1] = s[n][3] = -INFINITY;
      }
    }
    // Online softmax (base 2, scores pre-scaled by log2(e)/sqrt(hd)).
    float mx0 = m0, mx1 = m1;
#pragma unroll
    for (int n = 0; n < 8; ++n) {
      mx0 = fmaxf(mx0, fmaxf(s[n][0], s[n][1]) * sl2);
      mx1 = fmaxf(mx1, fmaxf(s[n][2], s[n][3]) * sl2);
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float c0 = exp2f(m0 - mx0), c1 = exp2f(m1 - mx1);  // 0 on the first tile (m = -inf)
    m0 = mx0;
    m1 = mx1;
    float rs0 = 0.f, rs1 = 0.f;
    uint32_t pa[4][4];  // P as A fragments, 4 k-steps of 16 keys
#pragma unroll
    for (int n = 0; n < 8; ++n) {
      const float p0 = exp2f(s[n][0] * sl2 - m0), p1 = exp2f(s[n][1] * sl2 - m0);
      const float p2 = exp2f(s[n][2] * sl2 - m1), p3 = exp2f(s[n][3] * sl2 - m1);
      rs0 += p0 + p1;
      rs1 += p2 + p3;
      pa[n >> 1][(n & 1) * 2 + 0] = pack_bf16x2(p0, p1);
      pa[n >> 1][(n & 1) * 2 + 1] = pack_bf16x2(p2, p3);
    }
    l0 = l0 * c0 + rs0;
    l1 = l1 * c1 + rs1;
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      o[i][0] *= c0;
      o[i][1] *= c0;
      o[i][2] *= c1;
      o[i][3] *= c1;
    }
    // O += P V.
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int dp = 0; dp < HD / 16; ++dp) {
        const int key = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int ch = dp * 2 + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(sv[buf] + swz<HD>(key, ch), b0, b1, b2, b3);
        mma_bf16_16816(o[2 * dp], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], b0, b1);
        mma_bf16_16816(o[2 * dp + 1], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], b2, b3);
      }
    }
    cp_async_wait<0>();
    __syncthreads();
  }

  // Row sums across the quad, normalise, store bf16.
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float inv0 = 1.f / l0, inv1 = 1.f / l1;
  const int g = lane >> 2, t = lane & 3;
  const int r0 = q0 + warp * 16 + g, r1 = r0 + 8;
  const int64_t ldo = static_cast<int64_t>(Hq) * HD;
  uint16_t* ob = out + (static_cast<int64_t>(b) * q_len - q_start) * ldo + static_cast<int64_t>(h) * HD;
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) {
    const int col = i * 8 + t * 2;
    if (r0 < q_end) *reinterpret_cast<uint32_t*>(ob + static_cast<int64_t>(r0) * ldo + col) = pack_bf16x2(o[i][0] * inv0, o[i][1] * inv0);
    if (r1 < q_end) *reinterpret_cast<uint32_t*>(ob + static_cast<int64_t>(r1) * ldo + col) = pack_bf16x2(o[i][2] * inv1, o[i][3] * inv1);
  }
}

}  // namespace cora

using namespace cora;

void launch_attention(const uint16_t* qkv, uint16_t* out, int B, int S, int Hq, int Hkv, int hd, int q_start,
                      int q_len, cudaStream_t st) {
  dim3 grid((q_len + kQT - 1) / kQT, Hq, B);
  const int smem = (kQT + 4 * kKT) * hd * 2;
  if (hd == 128)
    launch_pdl(attention_kernel<128>, grid, dim3(128), smem, st, qkv, out, S, Hq, Hkv, q_start, q_len);
  else
    launch_pdl(attention_kernel<64>, grid, dim3(128), smem, st, qkv, out, S, Hq, Hkv, q_start, q_len);
}

cudaError_t attention_prepare() {
  cudaError_t e = cudaFuncSetAttribute(attention_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (kQT + 4 * kKT) * 128 * 2);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attention_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (kQT + 4 * kKT) * 64 * 2);
}
