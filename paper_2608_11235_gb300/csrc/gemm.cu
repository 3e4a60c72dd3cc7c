// Dense bf16 GEMM on the 5th-generation tensor cores (tcgen05) for the
// backbone's projections: acc[M, N] = A[M, K] * B[N, K]^T, fp32 accumulation
// in TMEM, operands staged in shared memory by TMA with 128-byte swizzling.
//
// Persistent kernel, one CTA per SM, 6 warps:
//   warp 0      TMA producer (one elected lane): A and B K-slices into a ring
//               of STAGES shared-memory buffers (full/empty mbarriers);
//   warp 1      TMEM allocator and MMA issuer (one lane): 128 x BN x 16
//               tcgen05.mma per K step, tcgen05.commit frees ring slots;
//   warps 2..5  epilogue: tcgen05.ld of the 128 x BN accumulator (warp w
//               reads TMEM lanes 32*(w%4) .. +31, one output row per thread),
//               fused epilogue, global stores.
// Two TMEM accumulators (2 * BN columns) let the epilogue of tile i overlap
// the MMAs of tile i+1.  Tiles are visited M-fastest so the CTAs working at
// the same time share the weight tile (B) through L2.
#include <math.h>

#include "cora_device.cuh"
#include "cora_kernels.h"
#include "../../include/cora.h"

namespace cora {

constexpr int kBM = 128;
constexpr int kBK = 64;  // 64 bf16 = 128 bytes = one swizzle row

template <int BN>
struct GemmCfg {
  static constexpr int A_BYTES = kBM * kBK * 2;
  static constexpr int B_BYTES = BN * kBK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = BN == 256 ? 4 : 6;
  static constexpr int TMEM_COLS = 2 * BN;
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/;
};

__device__ __forceinline__ float silu_f(float x) { return x / (1.f + __expf(-x)); }

__device__ __forceinline__ void store_bf16x16(uint16_t* dst, const float (&v)[16]) {
  uint4 a, b;
  a.x = pack_bf16x2(v[0], v[1]);
  a.y = pack_bf16x2(v[2], v[3]);
  a.z = pack_bf16x2(v[4], v[5]);
  a.w = pack_bf16x2(v[6], v[7]);
  b.x = pack_bf16x2(v[8], v[9]);
  b.y = pack_bf16x2(v[10], v[11]);
  b.z = pack_bf16x2(v[12], v[13]);
  b.w = pack_bf16x2(v[14], v[15]);
  reinterpret_cast<uint4*>(dst)[0] = a;
  reinterpret_cast<uint4*>(dst)[1] = b;
}

// Epilogue of one 128 x BN tile for the calling thread's row.
template <int BN>
__device__ __forceinline__ void gemm_epilogue_row(const GemmEpilogue& ep, uint32_t tacc, int row, int M, int n0) {
  const bool in_range = row < M;
  if (ep.mode == CORA_EPI_STORE_BF16) {
    uint16_t* crow = reinterpret_cast<uint16_t*>(ep.C) + static_cast<int64_t>(row) * ep.ldc + n0;
#pragma unroll 1
    for (int c = 0; c < BN; c += 16) {
      float v[16];
      tmem_ld16(tacc + c, v);
      if (in_range) store_bf16x16(crow + c, v);
    }
  } else if (ep.mode == CORA_EPI_RESID_F32) {
    float* crow = reinterpret_cast<float*>(ep.C) + static_cast<int64_t>(row) * ep.ldc + n0;
#pragma unroll 1
    for (int c = 0; c < BN; c += 16) {
      float v[16];
      tmem_ld16(tacc + c, v);
      if (in_range) {
        float4* p = reinterpret_cast<float4*>(crow + c);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float4 h = p[q];
          h.x += v[4 * q];
          h.y += v[4 * q + 1];
          h.z += v[4 * q + 2];
          h.w += v[4 * q + 3];
          p[q] = h;
        }
      }
    }
  } else if (ep.mode == CORA_EPI_SWIGLU) {
    // Tile columns [0, BN/2) are gate rows, [BN/2, BN) the matching up rows
    // of output features n0/2 .. n0/2 + BN/2.
    uint16_t* crow = reinterpret_cast<uint16_t*>(ep.C) + static_cast<int64_t>(row) * ep.ldc + n0 / 2;
#pragma unroll 1
    for (int c = 0; c < BN / 2; c += 16) {
      float g[16], u[16];
      tmem_ld16x2(tacc + c, tacc + BN / 2 + c, g, u);
#pragma unroll
      for (int j = 0; j < 16; ++j) g[j] = silu_f(g[j]) * u[j];
      if (in_range) store_bf16x16(crow + c, g);
    }
  } else {  // CORA_EPI_ROPE_BF16
    uint16_t* crow = reinterpret_cast<uint16_t*>(ep.C) + static_cast<int64_t>(row) * ep.ldc + n0;
    const int hd = ep.head_dim, half = hd / 2;
    const int pos = in_range ? row % ep.seq : 0;
    const float2* tab = reinterpret_cast<const float2*>(ep.rope) + static_cast<int64_t>(pos) * half;
#pragma unroll 1
    for (int h0 = 0; h0 < BN; h0 += hd) {
      const bool rot = n0 + h0 < ep.rope_cols;
#pragma unroll 1
      for (int j0 = 0; j0 < half; j0 += 16) {
        float x1[16], x2[16];
        tmem_ld16x2(tacc + h0 + j0, tacc + h0 + half + j0, x1, x2);
        if (rot) {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float2 cs = tab[j0 + j];
            const float a = x1[j], b = x2[j];
            x1[j] = a * cs.x - b * cs.y;
            x2[j] = b * cs.x + a * cs.y;
          }
        }
        if (in_range) {
          store_bf16x16(crow + h0 + j0, x1);
          store_bf16x16(crow + h0 + half + j0, x2);
        }
      }
    }
  }
}

template <int BN>
__global__ void __launch_bounds__(192, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, int M, int N,
                   int K, GemmEpilogue ep, int* err) {
  using Cfg = GemmCfg<BN>;
  constexpr int STAGES = Cfg::STAGES;
  constexpr uint32_t IDESC = idesc_bf16_f32(kBM, BN);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * Cfg::STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_m = (M + kBM - 1) / kBM;
  const int num_tiles = num_m * (N / BN);
  const int kblocks = K / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 128);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
        const int mb = t % num_m, nb = t / num_m;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err, CORA_DERR_TMA_WAIT)) goto producer_done;
          uint8_t* sa = smem + stage * Cfg::STAGE_BYTES;
          mbar_arrive_expect_tx(&full[stage], Cfg::STAGE_BYTES);
          tma_load_2d(sa, &tmA, &full[stage], kb * kBK, mb * kBM);
          tma_load_2d(sa + Cfg::A_BYTES, &tmB, &full[stage], kb * kBK, nb * BN);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    producer_done:;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++it) {
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, err, CORA_DERR_MMA_WAIT)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        bool ok = true;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, err, CORA_DERR_MMA_WAIT)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = smem_u32(smem + stage * Cfg::STAGE_BYTES);
          const uint32_t b_addr = a_addr + Cfg::A_BYTES;
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            umma_bf16(d_tmem, sw128_kmajor_desc(a_addr + k * 32), sw128_kmajor_desc(b_addr + k * 32), IDESC,
                      (kb | k) != 0);
          }
          umma_commit(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
      }
    }
  } else {
    const int sub = warp & 3;  // TMEM sub-partition this warp may access
    int it = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++it) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      if (!mbar_wait(&tfull[acc], acc_phase, abort_flag, err, CORA_DERR_EPI_WAIT)) break;
      tc_fence_after();
      const int mb = t % num_m, nb = t / num_m;
      const int row = mb * kBM + sub * 32 + lane;
      const uint32_t tacc = tmem_base + (static_cast<uint32_t>(sub * 32) << 16) + acc * BN;
      gemm_epilogue_row<BN>(ep, tacc, row, M, nb * BN);
      tc_fence_before();
      mbar_arrive(&tempty[acc]);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
  }
}

}  // namespace cora

using namespace cora;

int gemm_block_n(int N, int mode) {
  if (mode == CORA_EPI_SWIGLU) return 256;
  return (N % 256 == 0) ? 256 : 128;
}

template <int BN>
static cudaError_t launch_gemm_bn(const CUtensorMap& tmA, const CUtensorMap& tmB, int M, int N, int K,
                                  const GemmEpilogue& ep, int* err, int num_sms, cudaStream_t st) {
  using Cfg = GemmCfg<BN>;
  const int tiles = ((M + kBM - 1) / kBM) * (N / BN);
  const int grid = tiles < num_sms ? tiles : num_sms;
  gemm_tc_kernel<BN><<<grid, 192, Cfg::SMEM_BYTES, st>>>(tmA, tmB, M, N, K, ep, err);
  return cudaGetLastError();
}

cudaError_t gemm_prepare() {
  cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       GemmCfg<256>::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(gemm_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              GemmCfg<128>::SMEM_BYTES);
}

cudaError_t launch_gemm(const CUtensorMap& tmA, const CUtensorMap& tmB, int M, int N, int K, const GemmEpilogue& ep,
                        int* err, int num_sms, cudaStream_t st) {
  if (gemm_block_n(N, ep.mode) == 256) return launch_gemm_bn<256>(tmA, tmB, M, N, K, ep, err, num_sms, st);
  return launch_gemm_bn<128>(tmA, tmB, M, N, K, ep, err, num_sms, st);
}
