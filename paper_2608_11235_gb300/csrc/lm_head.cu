// Fused LM head + Eq. 1 (top-1 confidence and prediction) for the active
// block's rows only.  The logits [R, V] never reach memory: each 128-wide
// vocabulary tile is computed on the tensor cores as D[128 vocab, NPAD rows]
// = W[v0:v0+128, :] * X^T (swap-AB: the long vocabulary axis fills the
// M = 128 side, the few active rows sit on N), and the epilogue reduces it
// straight out of TMEM into per-row running (max, sum exp, argmax) states.
// Each persistent CTA writes one partial per row; the gate kernel combines
// the partials in CTA order (deterministic, lowest id wins ties).
//
// Work per launch is streaming the head (V * d * 2 bytes) once: an HBM-bound
// kernel for R <= ~128 rows.
#include <limits.h>
#include <math.h>

#include "cora_device.cuh"
#include "cora_kernels.h"

namespace cora {

constexpr int kVT = 128;  // vocabulary rows per tile (MMA M)
constexpr int kKB = 64;   // K per stage (one 128-byte swizzle row)

template <int NPAD>
struct HeadCfg {
  static constexpr int A_BYTES = kVT * kKB * 2;
  static constexpr int B_BYTES = NPAD * kKB * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES_RAW = (180 * 1024) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_RAW > 12 ? 12 : STAGES_RAW;
  static constexpr int TMEM_COLS = 2 * NPAD < 32 ? 32 : 2 * NPAD;
  static constexpr int RED_BYTES = 5 * NPAD * 12;  // 4 warp partials + running state
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256 + RED_BYTES;
};

template <int NPAD>
__global__ void __launch_bounds__(192, 1)
    lm_head_top1_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX, int R,
                        int V, int d, Top1Part* __restrict__ parts, int* err) {
  using Cfg = HeadCfg<NPAD>;
  constexpr int STAGES = Cfg::STAGES;
  constexpr uint32_t IDESC = idesc_bf16_f32(kVT, NPAD);
  constexpr float kLog2e = 1.4426950408889634f;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * Cfg::STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  Top1* wpart = reinterpret_cast<Top1*>(smem + STAGES * Cfg::STAGE_BYTES + 256);  // [4][NPAD]
  Top1* run = wpart + 4 * NPAD;                                                   // [NPAD]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_tiles = (V + kVT - 1) / kVT;
  const int kblocks = d / kKB;

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
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    tmem_relinquish();
  }
  __syncwarp();  // converged arrival (one lane of warp 0 initialised the barriers)
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_trigger();
  pdl_wait();  // the normalised rows come from the previous kernel

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t stream_w = l2_policy_evict_first();  // the head is read once per launch
      const uint64_t keep_x = l2_policy_evict_last();     // the rows are re-read by every tile
      int stage = 0;
      uint32_t phase = 0;
      for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err, CORA_DERR_TMA_WAIT)) goto producer_done;
          uint8_t* sa = smem + stage * Cfg::STAGE_BYTES;
          mbar_arrive_expect_tx(&full[stage], Cfg::STAGE_BYTES);
          tma_load_2d_hint(sa, &tmW, &full[stage], kb * kKB, t * kVT, stream_w);
          tma_load_2d_hint(sa + Cfg::A_BYTES, &tmX, &full[stage], kb * kKB, 0, keep_x);
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
        const uint32_t d_tmem = tmem_base + acc * NPAD;
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
          for (int k = 0; k < kKB / 16; ++k) {
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
    const int sub = warp & 3;
    const int etid = threadIdx.x - 64;  // 0..127
    for (int r = etid; r < NPAD; r += 128) run[r] = Top1{-INFINITY, 0.f, INT_MAX};
    named_bar_sync(1, 128);
    int it = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++it) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const bool ok = mbar_wait(&tfull[acc], acc_phase, abort_flag, err, CORA_DERR_EPI_WAIT);
      if (ok) {
      tc_fence_after();
      const int v = t * kVT + sub * 32 + lane;  // this thread's vocabulary id
      const bool valid = v < V;
      const uint32_t tacc = tmem_base + (static_cast<uint32_t>(sub * 32) << 16) + acc * NPAD;
#pragma unroll 1
      for (int c = 0; c < NPAD; c += 16) {
        float x[16];
        tmem_ld16(tacc + c, x);
#pragma unroll 4
        for (int j = 0; j < 16; ++j) {
          float m = valid ? x[j] : -INFINITY;
          int id = valid ? v : INT_MAX;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
            const float om = __shfl_xor_sync(0xffffffffu, m, o);
            const int oi = __shfl_xor_sync(0xffffffffu, id, o);
            if (om > m || (om == m && oi < id)) {
              m = om;
              id = oi;
            }
          }
          float e = valid ? exp2f((x[j] - m) * kLog2e) : 0.f;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) e += __shfl_xor_sync(0xffffffffu, e, o);
          if (lane == 0) wpart[sub * NPAD + c + j] = Top1{m, e, id};
        }
      }
      tc_fence_before();
      mbar_arrive(&tempty[acc]);
      }
      // Uniform exit: every epilogue warp leaves together if any wait failed.
      if (named_bar_or(1, 128, !ok)) break;
      for (int r = etid; r < NPAD; r += 128) {
        Top1 st = run[r];
#pragma unroll
        for (int w = 0; w < 4; ++w) st = top1_merge(st, wpart[w * NPAD + r]);
        run[r] = st;
      }
      named_bar_sync(1, 128);
    }
    for (int r = etid; r < R; r += 128) {
      const Top1 st = run[r];
      parts[static_cast<int64_t>(blockIdx.x) * R + r] = Top1Part{st.m, st.s, st.idx};
    }
  }

  // Each warp arrives converged: the producer and MMA warps ran their loops
  // on one lane, and bar.sync counts a divergent warp's lanes separately.
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
  }
}

}  // namespace cora

using namespace cora;

int lm_head_npad(int R) {
  if (R <= 16) return 16;
  if (R <= 32) return 32;
  if (R <= 64) return 64;
  if (R <= 128) return 128;
  return 256;
}

int lm_head_parts_count(int V, int num_sms) {
  const int tiles = (V + kVT - 1) / kVT;
  return tiles < num_sms ? tiles : num_sms;
}

template <int NPAD>
static cudaError_t launch_head_n(const CUtensorMap& tmW, const CUtensorMap& tmX, int R, int V, int d,
                                 Top1Part* parts, int n_parts, int* err, cudaStream_t st) {
  using Cfg = HeadCfg<NPAD>;
  launch_pdl(lm_head_top1_kernel<NPAD>, dim3(n_parts), dim3(192), Cfg::SMEM_BYTES, st, tmW, tmX, R, V, d, parts, err);
  return cudaGetLastError();
}

template <int NPAD>
static cudaError_t prepare_head_n() {
  return cudaFuncSetAttribute(lm_head_top1_kernel<NPAD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              HeadCfg<NPAD>::SMEM_BYTES);
}

cudaError_t lm_head_prepare() {
  cudaError_t e;
  if ((e = prepare_head_n<16>()) != cudaSuccess) return e;
  if ((e = prepare_head_n<32>()) != cudaSuccess) return e;
  if ((e = prepare_head_n<64>()) != cudaSuccess) return e;
  if ((e = prepare_head_n<128>()) != cudaSuccess) return e;
  return prepare_head_n<256>();
}

cudaError_t launch_lm_head_top1(const CUtensorMap& tmW, const CUtensorMap& tmX, int R, int V, int d,
                                Top1Part* parts, int n_parts, int* err, cudaStream_t st) {
  switch (lm_head_npad(R)) {
    case 16: return launch_head_n<16>(tmW, tmX, R, V, d, parts, n_parts, err, st);
    case 32: return launch_head_n<32>(tmW, tmX, R, V, d, parts, n_parts, err, st);
    case 64: return launch_head_n<64>(tmW, tmX, R, V, d, parts, n_parts, err, st);
    case 128: return launch_head_n<128>(tmW, tmX, R, V, d, parts, n_parts, err, st);
    default: return launch_head_n<256>(tmW, tmX, R, V, d, parts, n_parts, err, st);
  }
}
