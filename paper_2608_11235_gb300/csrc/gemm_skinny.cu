// Few-row GEMM (M <= 64 activation rows) on the 5th-generation tensor
// cores, swap-AB: D[n, m] = sum_k W[n, k] X[m, k] with the weight rows n on
// the MMA's M = 128 side and the activation rows m on N (padded to NPAD), so
// each CTA streams its slice of the weights once while the few activation
// rows are re-read from L2.  For these shapes the work is streaming the
// weights (N * K * 2 bytes per launch): an HBM-bound kernel, where the
// row-tiled kernel would pad the rows to 128 and split tiles over k.
//
// Tiles are TR = 128 weight rows (TR = 256 for SwiGLU: the gate group and
// its up group, two accumulators).  Work split: units (tile, piece), each
// tile cut into S equal k-ranges (S = 1 when there are enough tiles to fill
// the GPU), CTAs taking units round-robin.  A tile cut into S > 1 pieces is
// finished by the LAST piece to arrive (a ticket per tile), which adds every
// piece's fp32 partial in piece order (deterministic; no CTA waits on
// another) and runs the epilogue.
//
// Epilogues act on the transposed accumulator: an epilogue thread owns one
// weight row n (TMEM lane) and loops over the activation rows m:
//   STORE   C[m][n] = bf16(d)                   (coalesced along n)
//   RESID   C[m][n] += d (fp32 residual stream; the finisher is the only
//           writer of its tile, so a plain read-add-write is exact)
//   ROPE    rotate-half pairs (n, n ^ hd/2) exchanged through shared memory
//   SWIGLU  C[m][f] = bf16(silu(gate) * up), gate and up from the two accumulators
// With out3d, row m goes to sequence m / seq, position rope_pos0 + m % seq
// (the packed rows of a prefix-cache pass).
//
// Warps: 0 = TMA producer, 1 = TMEM allocator + MMA issuer, 2..5 = epilogue.
#include <math.h>

#include "cora_device.cuh"
#include "cora_kernels.h"
#include "../../include/cora.h"

namespace cora {

namespace sk {
constexpr int KB = 64;           // K per stage (one 128-byte swizzle row)
constexpr int TICKETS = 512;     // ticket counters live at ws.flags + TICKETS (after the row-tiled kernel's flags)
constexpr int MAX_PIECES = 4;
}  // namespace sk

template <int NPAD, int TR>
struct SkCfg {
  static constexpr int W_BYTES = TR * sk::KB * 2;
  static constexpr int X_BYTES = NPAD * sk::KB * 2;
  static constexpr int STAGE_BYTES = W_BYTES + X_BYTES;
  static constexpr int STAGES_RAW = (176 * 1024) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_RAW > 12 ? 12 : STAGES_RAW;
  static constexpr int ACC_COLS = (TR / 128) * NPAD;  // one accumulator set
  static constexpr int NBUF = 2 * ACC_COLS <= 512 ? 2 : 1;
  static constexpr int COLS_USED = NBUF * ACC_COLS;
  static constexpr int TMEM_COLS = COLS_USED <= 32 ? 32 : COLS_USED <= 64 ? 64 : COLS_USED <= 128 ? 128
                                   : COLS_USED <= 256 ? 256 : 512;
  static constexpr int EX_BYTES = 128 * 16 * 4;  // RoPE exchange: 128 rows x 16 columns fp32
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256 + EX_BYTES;
};

// Partial slot layout: [NPAD/4][TR][4] fp32, so a warp's float4 access over
// its 32 consecutive rows covers 512 contiguous bytes.
__device__ __forceinline__ int64_t sk_f4(int m, int n, int tr) { return static_cast<int64_t>(m >> 2) * tr + n; }

// silu as in the row-tiled kernels (approximate divide, bf16 result)
__device__ __forceinline__ float silu_sk(float x) { return __fdividef(x, 1.f + __expf(-x)); }

template <int NPAD, int TR>
__global__ void __launch_bounds__(192, 1)
    gemm_skinny_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX, int M, int N,
                       int K, int S, GemmEpilogue ep, GemmWorkspace ws, int* err) {
  using Cfg = SkCfg<NPAD, TR>;
  constexpr int STAGES = Cfg::STAGES;
  constexpr uint32_t IDESC = idesc_bf16_f32(128, NPAD);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * Cfg::STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* last_flag = const_cast<int*>(reinterpret_cast<volatile int*>(abort_flag + 1));
  float* ex = reinterpret_cast<float*>(smem + STAGES * Cfg::STAGE_BYTES + 256);  // [128][16]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tiles = N / TR;
  const int KBn = K / sk::KB;
  const int units = tiles * S;
  // unit u: tile u / S, k-blocks [p KBn / S, (p+1) KBn / S) with p = u % S
  auto unit_range = [&](int u, int& t, int& kb0, int& kb1) {
    t = u / S;
    const int p = u - t * S;
    kb0 = p * KBn / S;
    kb1 = (p + 1) * KBn / S;
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 4);
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
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t stream_w = l2_policy_evict_first();  // the weights are read once per launch
      const uint64_t keep_x = l2_policy_evict_last();     // the rows are re-read by every tile
      int stage = 0;
      uint32_t phase = 0;
      for (int u = blockIdx.x; u < units; u += gridDim.x) {
        int t, kb0, kb1;
        unit_range(u, t, kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err, CORA_DERR_TMA_WAIT)) goto producer_done;
          uint8_t* sa = smem + stage * Cfg::STAGE_BYTES;
          mbar_arrive_expect_tx(&full[stage], Cfg::STAGE_BYTES);
#pragma unroll
          for (int h = 0; h < TR / 128; ++h)
            tma_load_2d_hint(sa + h * 128 * sk::KB * 2, &tmW, &full[stage], kb * sk::KB, t * TR + h * 128, stream_w);
          tma_load_2d_hint(sa + Cfg::W_BYTES, &tmX, &full[stage], kb * sk::KB, 0, keep_x);
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
      for (int u = blockIdx.x; u < units; u += gridDim.x, ++it) {
        int t, kb0, kb1;
        unit_range(u, t, kb0, kb1);
        const int buf = Cfg::NBUF == 2 ? (it & 1) : 0;
        const uint32_t buf_phase = Cfg::NBUF == 2 ? ((it >> 1) & 1) : (it & 1);
        if (!mbar_wait(&tempty[buf], buf_phase ^ 1u, abort_flag, err, CORA_DERR_MMA_WAIT)) break;
        tc_fence_after();
        const uint32_t d0 = tmem_base + buf * Cfg::ACC_COLS;
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, err, CORA_DERR_MMA_WAIT)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t w_addr = smem_u32(smem + stage * Cfg::STAGE_BYTES);
          const uint32_t x_addr = w_addr + Cfg::W_BYTES;
#pragma unroll
          for (int k = 0; k < sk::KB / 16; ++k) {
#pragma unroll
            for (int h = 0; h < TR / 128; ++h)
              umma_bf16(d0 + h * NPAD, sw128_kmajor_desc(w_addr + h * 128 * sk::KB * 2 + k * 32),
                        sw128_kmajor_desc(x_addr + k * 32), IDESC, (kb > kb0 || k > 0) ? 1u : 0u);
          }
          umma_commit(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(&tfull[buf]);
      }
    }
  } else {
    const int sub = warp & 3;
    const int etid = threadIdx.x - 64;
    const int nl = sub * 32 + lane;  // row of the tile (TMEM lane) in each 128-row accumulator
    const int hd = ep.head_dim, half = hd / 2;
    int it = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++it) {
      int t, kb0, kb1;
      unit_range(u, t, kb0, kb1);
      const int buf = Cfg::NBUF == 2 ? (it & 1) : 0;
      const uint32_t buf_phase = Cfg::NBUF == 2 ? ((it >> 1) & 1) : (it & 1);
      const bool ok = mbar_wait(&tfull[buf], buf_phase, abort_flag, err, CORA_DERR_EPI_WAIT);
      if (named_bar_or(1, 128, !ok)) break;
      tc_fence_after();
      const uint32_t tacc = tmem_base + (static_cast<uint32_t>(sub * 32) << 16) + buf * Cfg::ACC_COLS;
      const bool whole = S == 1;
      const int slot_me = u;  // partial slot of this piece
      // ---- split tile: hand the partial in, the last arriver finishes
      if (!whole) {
        float4* dst = reinterpret_cast<float4*>(ws.partial) + static_cast<int64_t>(slot_me) * (TR * NPAD / 4);
#pragma unroll 1
        for (int m0 = 0; m0 < NPAD; m0 += 16) {
#pragma unroll
          for (int h = 0; h < TR / 128; ++h) {
            float v[16];
            tmem_ld16(tacc + h * NPAD + m0, v);
#pragma unroll
            for (int q = 0; q < 4; ++q)
              dst[sk_f4(m0 + 4 * q, h * 128 + nl, TR)] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[buf]);
        __threadfence();
        named_bar_sync(1, 128);
        if (etid == 0) {
          const int old = atomicAdd(ws.flags + sk::TICKETS + t, 1);
          *last_flag = old == S - 1;
          if (*last_flag) atomicExch(ws.flags + sk::TICKETS + t, 0);  // ready for the next launch
        }
        named_bar_sync(1, 128);
        if (!*last_flag) continue;
        __threadfence();  // acquire: every other piece's partial is visible
      }
      // ---- epilogue over the activation rows, 16 at a time
      const int64_t n_glob = static_cast<int64_t>(t) * (TR == 256 ? 128 : TR) + nl;  // output column (SwiGLU: feature)
#pragma unroll 1
      for (int m0 = 0; m0 < NPAD; m0 += 16) {
        float v[TR / 128][16];
        if (whole) {
#pragma unroll
          for (int h = 0; h < TR / 128; ++h) tmem_ld16(tacc + h * NPAD + m0, v[h]);
        } else {
          // every piece's 16 columns loaded before any is added (one memory
          // round trip per chunk), then summed in piece order
          float4 xs[sk::MAX_PIECES][TR / 128][4];
#pragma unroll
          for (int p = 0; p < sk::MAX_PIECES; ++p) {
            if (p < S) {
              const float4* src =
                  reinterpret_cast<const float4*>(ws.partial) + static_cast<int64_t>(t * S + p) * (TR * NPAD / 4);
#pragma unroll
              for (int h = 0; h < TR / 128; ++h)
#pragma unroll
                for (int q = 0; q < 4; ++q) xs[p][h][q] = __ldcg(src + sk_f4(m0 + 4 * q, h * 128 + nl, TR));
            }
          }
#pragma unroll
          for (int h = 0; h < TR / 128; ++h)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              float4 a = xs[0][h][q];
#pragma unroll
              for (int p = 1; p < sk::MAX_PIECES; ++p)
                if (p < S) {
                  a.x += xs[p][h][q].x;
                  a.y += xs[p][h][q].y;
                  a.z += xs[p][h][q].z;
                  a.w += xs[p][h][q].w;
                }
              v[h][4 * q] = a.x;
              v[h][4 * q + 1] = a.y;
              v[h][4 * q + 2] = a.z;
              v[h][4 * q + 3] = a.w;
            }
        }
        if (ep.mode == CORA_EPI_RESID_F32) {
          // all 16 residuals loaded before any store: one memory round trip
          // per chunk instead of a chain of 16 read-add-writes
          float* C = static_cast<float*>(ep.C);
          float res[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int m = m0 + j;
            res[j] = m < M ? __ldcg(C + static_cast<int64_t>(m) * ep.ldc + n_glob) : 0.f;
          }
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int m = m0 + j;
            if (m < M) C[static_cast<int64_t>(m) * ep.ldc + n_glob] = res[j] + v[0][j];
          }
        } else if (ep.mode == CORA_EPI_SWIGLU) {
          uint16_t* C = static_cast<uint16_t*>(ep.C);
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int m = m0 + j;
            if (m < M) {
              const float g = v[0][j], u = v[TR / 128 - 1][j];
              C[static_cast<int64_t>(m) * ep.ldc + n_glob] =
                  static_cast<uint16_t>(pack_bf16x2(silu_sk(g) * u, 0.f) & 0xFFFFu);
            }
          }
        } else {
          const bool rope = ep.mode == CORA_EPI_ROPE_BF16 && n_glob < ep.rope_cols;
          if (ep.mode == CORA_EPI_ROPE_BF16) {
            // partner row of the rotate-half pair (tile rows are head-aligned)
#pragma unroll
            for (int j = 0; j < 16; ++j) ex[nl * 16 + ((j + lane) & 15)] = v[0][j];
            named_bar_sync(1, 128);
            const int pn = nl ^ half;
            const int jj = static_cast<int>(n_glob % hd);
            // the chunk's 16 (cos, sin) pairs loaded together, ahead of their use
            float2 cs[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int m = m0 + j;
              cs[j] = rope && m < M ? __ldg(reinterpret_cast<const float2*>(ep.rope) +
                                            static_cast<int64_t>(ep.rope_pos0 + m % ep.seq) * half + (jj % half))
                                    : make_float2(1.f, 0.f);
            }
            float r[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float other = ex[pn * 16 + ((j + (pn & 31)) & 15)];
              r[j] = !rope ? v[0][j]
                     : jj < half ? v[0][j] * cs[j].x - other * cs[j].y
                                 : v[0][j] * cs[j].x + other * cs[j].y;
            }
            named_bar_sync(1, 128);  // ex is rewritten by the next chunk
#pragma unroll
            for (int j = 0; j < 16; ++j) v[0][j] = r[j];
          }
          uint16_t* C = static_cast<uint16_t*>(ep.C);
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int m = m0 + j;
            if (m < M) {
              const int64_t row = ep.out3d ? static_cast<int64_t>(m / ep.seq) * ep.out_rows_per_seq + ep.rope_pos0 +
                                                 m % ep.seq
                                           : m;
              C[row * ep.ldc + n_glob] = static_cast<uint16_t>(pack_bf16x2(v[0][j], 0.f) & 0xFFFFu);
            }
          }
        }
      }
      if (whole) {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[buf]);
      }
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

template <int NPAD, int TR>
static cudaError_t launch_sk(const CUtensorMap& tmW, const CUtensorMap& tmX, int M, int N, int K,
                             const GemmEpilogue& ep, const GemmWorkspace& ws, int* err, int num_sms, cudaStream_t st) {
  using Cfg = SkCfg<NPAD, TR>;
  static bool prepared = false;
  if (!prepared) {
    cudaError_t e = cudaFuncSetAttribute(gemm_skinny_kernel<NPAD, TR>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Cfg::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    prepared = true;
  }
  const int tiles = N / TR, KBn = K / sk::KB;
  // Whole tiles when they nearly fill the GPU; otherwise up to MAX_PIECES
  // equal k-pieces per tile (each at least four k-blocks).
  int S = 1;
  if (2 * tiles < num_sms) {
    S = num_sms / tiles;
    if (S > sk::MAX_PIECES) S = sk::MAX_PIECES;
    if (S > KBn / 4) S = KBn / 4;
    if (S < 1) S = 1;
  }
  const int units = tiles * S;
  if (S > 1 && static_cast<size_t>(units) * TR * NPAD * sizeof(float) > gemm_workspace_bytes(num_sms))
    return cudaErrorInvalidValue;
  const int G = units < num_sms ? units : num_sms;
  return launch_pdl(gemm_skinny_kernel<NPAD, TR>, dim3(G), dim3(192), Cfg::SMEM_BYTES, st, tmW, tmX, M, N, K, S, ep,
                    ws, err);
}

}  // namespace cora

using namespace cora;

int gemm_skinny_npad(int M) { return M <= 16 ? 16 : M <= 32 ? 32 : 64; }

bool gemm_skinny_supported(int M, int N, int K, const GemmEpilogue& ep) {
  // Measured on the LLaDA-8B shapes: faster than the row-tiled kernel up to
  // 64 rows, slower from 96 on (the rows' re-reads grow with NPAD).
  if (M < 1 || M > 64 || !ep.a_ptr || K % sk::KB != 0) return false;
  const int TR = ep.mode == CORA_EPI_SWIGLU ? 256 : 128;
  if (N % TR != 0 || N / TR > sk::TICKETS) return false;
  if (ep.mode == CORA_EPI_ROPE_BF16 && (ep.head_dim > 128 || 128 % ep.head_dim != 0)) return false;
  return true;
}

cudaError_t launch_gemm_skinny(const CUtensorMap& tmW, const CUtensorMap& tmX, int M, int N, int K,
                               const GemmEpilogue& ep, const GemmWorkspace& ws, int* err, int num_sms,
                               cudaStream_t st) {
  const bool sw = ep.mode == CORA_EPI_SWIGLU;
  switch (gemm_skinny_npad(M)) {
    case 16: return sw ? launch_sk<16, 256>(tmW, tmX, M, N, K, ep, ws, err, num_sms, st)
                       : launch_sk<16, 128>(tmW, tmX, M, N, K, ep, ws, err, num_sms, st);
    case 32: return sw ? launch_sk<32, 256>(tmW, tmX, M, N, K, ep, ws, err, num_sms, st)
                       : launch_sk<32, 128>(tmW, tmX, M, N, K, ep, ws, err, num_sms, st);
    default: return sw ? launch_sk<64, 256>(tmW, tmX, M, N, K, ep, ws, err, num_sms, st)
                       : launch_sk<64, 128>(tmW, tmX, M, N, K, ep, ws, err, num_sms, st);
  }
}
