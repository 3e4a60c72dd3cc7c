// Bidirectional (non-causal) attention on the 5th-generation tensor cores,
// head_dim 128.  One CTA per (sequence, query head, 128-query tile); keys and
// values stream through shared memory in 128-key tiles (TMA, double-buffered).
//
// Per key tile j:
//   S_j = Q K_j^T        tcgen05.mma M=128 (queries) x N=128 (keys) x K=128 (hd), TMEM
//   softmax              warps 2..5, one query row per thread: running max m and
//                        sum l (base 2, scores pre-scaled by log2(e)/sqrt(hd)),
//                        P_j = exp2(S_j - m_j) written to shared memory as bf16
//   O_j' = P_j V_j       tcgen05.mma M=128 x N=128 (hd) x K=128 (keys), V read as an
//                        MN-major operand straight from its [keys][hd] layout
//   O = a_j O + O_j'     in registers (a_j = exp2(m_{j-1} - m_j)), one row per thread
// Two TMEM buffers each for S and O' (512 columns) and two P buffers let the
// softmax of tile j overlap the MMAs of tiles j-1 and j+1.
// Warps: 0 = TMA producer, 1 = TMEM allocator + MMA issuer, 2..5 = softmax.
// Keys beyond the sequence end are masked; queries beyond it are not stored.
#include <math.h>

#include "cora_device.cuh"
#include "cora_kernels.h"

namespace cora {

namespace attn {
constexpr int QT = 128;          // queries per CTA
constexpr int KT = 128;          // keys per tile
constexpr int HD = 128;          // head dim
constexpr int OPND = QT * HD * 2;  // 32 KB: one 128 x 128 bf16 operand (two 16 KB swizzle columns)
constexpr int SMEM = 7 * OPND + 1024 + 256;  // Q, K[2], V[2], P[2]
}  // namespace attn

// MN-major (N contiguous) 128-byte-swizzled operand: 8-row K groups 1024 B
// apart (stride byte offset), 64-element N blocks `lbo` bytes apart.
__device__ __forceinline__ uint64_t sw128_mnmajor_desc(uint32_t smem_addr, uint32_t lbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((smem_addr & 0x3FFFF) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFF) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  float a[16], b[16];
  tmem_ld16x2(taddr, taddr + 16, a, b);
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    v[i] = a[i];
    v[16 + i] = b[i];
  }
}

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__global__ void __launch_bounds__(192, 1)
    attention_tc_kernel(const __grid_constant__ CUtensorMap tmQKV, uint16_t* __restrict__ out, int S, int Hq, int Hkv,
                        int* err) {
  using namespace attn;
  // idesc: M = 128, N = 128, bf16 x bf16 -> f32; PV reads B (V) MN-major.
  constexpr uint32_t IDESC_QK = idesc_bf16_f32(128, 128);
  constexpr uint32_t IDESC_PV = idesc_bf16_f32(128, 128) | (1u << 16);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK[2] = {smem + OPND, smem + 2 * OPND};
  uint8_t* sV[2] = {smem + 3 * OPND, smem + 4 * OPND};
  uint8_t* sP[2] = {smem + 5 * OPND, smem + 6 * OPND};
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 7 * OPND);
  uint64_t* qfull = bars + 0;
  uint64_t* kvfull = bars + 1;   // [2]
  uint64_t* kvempty = bars + 3;  // [2]
  uint64_t* sfull = bars + 5;    // [2]
  uint64_t* sfree = bars + 7;    // [2]
  uint64_t* pfull = bars + 9;    // [2]
  uint64_t* pfree = bars + 11;   // [2]
  uint64_t* ofull = bars + 13;   // [2]
  uint64_t* ofree = bars + 15;   // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 17);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int kvh = h / (Hq / Hkv);
  const int q0 = qt * QT;
  const int row_base = b * S;                       // first row of this sequence in [B*S, .]
  const int n_kt = (S + KT - 1) / KT;
  const int qcol = h * HD, kcol = (Hq + kvh) * HD, vcol = (Hq + Hkv + kvh) * HD;

  if (threadIdx.x == 0) {
    mbar_init(qfull, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kvfull[i], 1);
      mbar_init(&kvempty[i], 1);
      mbar_init(&sfull[i], 1);
      mbar_init(&sfree[i], 4);
      mbar_init(&pfull[i], 4);
      mbar_init(&pfree[i], 1);
      mbar_init(&ofull[i], 1);
      mbar_init(&ofree[i], 4);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) tma_prefetch_desc(&tmQKV);
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;  // S[0] at +0, S[1] at +128, O'[0] at +256, O'[1] at +384
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      mbar_arrive_expect_tx(qfull, OPND);
      tma_load_2d(sQ, &tmQKV, qfull, qcol, row_base + q0);
      tma_load_2d(sQ + OPND / 2, &tmQKV, qfull, qcol + 64, row_base + q0);
      for (int j = 0; j < n_kt; ++j) {
        const int s = j & 1;
        if (!mbar_wait(&kvempty[s], ((j >> 1) & 1) ^ 1u, abort_flag, err, CORA_DERR_TMA_WAIT)) break;
        mbar_arrive_expect_tx(&kvfull[s], 2 * OPND);
        const int r = row_base + j * KT;
        tma_load_2d(sK[s], &tmQKV, &kvfull[s], kcol, r);
        tma_load_2d(sK[s] + OPND / 2, &tmQKV, &kvfull[s], kcol + 64, r);
        tma_load_2d(sV[s], &tmQKV, &kvfull[s], vcol, r);
        tma_load_2d(sV[s] + OPND / 2, &tmQKV, &kvfull[s], vcol + 64, r);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = mbar_wait(qfull, 0, abort_flag, err, CORA_DERR_MMA_WAIT);
      const uint32_t q_addr = smem_u32(sQ);
      // PV of tile jj: O'[jj%2] = P[jj%2] V[jj%2].
      auto issue_pv = [&](int jj) -> bool {
        const int s = jj & 1;
        const uint32_t ph = (jj >> 1) & 1;
        if (!mbar_wait(&pfull[s], ph, abort_flag, err, CORA_DERR_MMA_WAIT)) return false;
        if (!mbar_wait(&ofree[s], ph ^ 1u, abort_flag, err, CORA_DERR_MMA_WAIT)) return false;
        tc_fence_after();
        const uint32_t p_addr = smem_u32(sP[s]), v_addr = smem_u32(sV[s]);
        const uint32_t d = tmem_base + 256 + s * 128;
#pragma unroll
        for (int k = 0; k < KT / 16; ++k) {
          // A = P: K-major, keys contiguous, 64-key swizzle columns 16 KB apart.
          const uint64_t a = sw128_kmajor_desc(p_addr + (k >> 2) * (OPND / 2) + (k & 3) * 32);
          // B = V: rows are keys (K), 64-element hd blocks 16 KB apart (MN-major).
          const uint64_t bd = sw128_mnmajor_desc(v_addr + k * 16 * 128, OPND / 2);
          umma_bf16(d, a, bd, IDESC_PV, k > 0);
        }
        umma_commit(&ofull[s]);
        umma_commit(&pfree[s]);
        umma_commit(&kvempty[s]);
        return true;
      };
      for (int j = 0; ok && j < n_kt; ++j) {
        const int s = j & 1;
        const uint32_t ph = (j >> 1) & 1;
        if (!mbar_wait(&kvfull[s], ph, abort_flag, err, CORA_DERR_MMA_WAIT)) break;
        if (!mbar_wait(&sfree[s], ph ^ 1u, abort_flag, err, CORA_DERR_MMA_WAIT)) break;
        tc_fence_after();
        const uint32_t k_addr = smem_u32(sK[s]);
        const uint32_t d = tmem_base + s * 128;
#pragma unroll
        for (int k = 0; k < HD / 16; ++k) {
          const uint32_t off = (k >> 2) * (OPND / 2) + (k & 3) * 32;
          umma_bf16(d, sw128_kmajor_desc(q_addr + off), sw128_kmajor_desc(k_addr + off), IDESC_QK, k > 0);
        }
        umma_commit(&sfull[s]);
        if (j >= 1 && !issue_pv(j - 1)) break;
      }
      if (ok && n_kt >= 1) issue_pv(n_kt - 1);
    }
  } else {
    const int sub = warp & 3;
    const int r = sub * 32 + lane;  // query row within the tile (TMEM lane)
    const uint32_t lane_base = tmem_base + (static_cast<uint32_t>(sub * 32) << 16);
    const float sl2 = 1.4426950408889634f / sqrtf(static_cast<float>(HD));
    float o[HD];
#pragma unroll
    for (int i = 0; i < HD; ++i) o[i] = 0.f;
    float m = -INFINITY, l = 0.f, a_prev = 1.f;
    bool ok = true;
    for (int j = 0; j <= n_kt && ok; ++j) {
      if (j < n_kt) {
        const int s = j & 1;
        const uint32_t ph = (j >> 1) & 1;
        ok = mbar_wait(&sfull[s], ph, abort_flag, err, CORA_DERR_EPI_WAIT);
        if (!ok) break;
        tc_fence_after();
        const uint32_t sb = lane_base + s * 128;
        const int kbase = j * KT;
        // pass 1: row max
        float mx = m;
#pragma unroll 1
        for (int c = 0; c < KT; c += 32) {
          float v[32];
          tmem_ld32(sb + c, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float x = (kbase + c + i < S) ? v[i] * sl2 : -INFINITY;
            mx = fmaxf(mx, x);
          }
        }
        const float alpha = ex2f(m - mx);  // 0 on the first tile (m = -inf)
        m = mx;
        // P buffer s is free once the PV of tile j-2 has read it.
        if (j >= 2) ok = mbar_wait(&pfree[s], ph ^ 1u, abort_flag, err, CORA_DERR_EPI_WAIT);
        if (!ok) break;
        // pass 2: P = exp2(S - m) as bf16 into the K-major swizzled P tile
        float rs = 0.f;
        uint8_t* prow = sP[s];
#pragma unroll 1
        for (int c = 0; c < KT; c += 32) {
          float v[32];
          tmem_ld32(sb + c, v);
          uint32_t pk[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float x0 = (kbase + c + 2 * i < S) ? ex2f(fmaf(v[2 * i], sl2, -m)) : 0.f;
            const float x1 = (kbase + c + 2 * i + 1 < S) ? ex2f(fmaf(v[2 * i + 1], sl2, -m)) : 0.f;
            rs += x0 + x1;
            pk[i] = pack_bf16x2(x0, x1);
          }
          // keys c .. c+31 -> swizzle column c/64, 16-byte chunks (c%64)/8 .. +3
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int key = c + 8 * q;
            const int chunk = (key & 63) >> 3;
            uint8_t* dst = prow + (key >> 6) * (OPND / 2) + r * 128 + ((chunk ^ (r & 7)) << 4);
            *reinterpret_cast<uint4*>(dst) = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
          }
        }
        l = l * alpha + rs;
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&sfree[s]);
          mbar_arrive(&pfull[s]);
        }
        // fold O'_{j-1} (computed with the previous max) into the row
        if (j >= 1) {
          const int sp = (j - 1) & 1;
          const uint32_t php = ((j - 1) >> 1) & 1;
          ok = mbar_wait(&ofull[sp], php, abort_flag, err, CORA_DERR_EPI_WAIT);
          if (!ok) break;
          tc_fence_after();
          const uint32_t ob = lane_base + 256 + sp * 128;
#pragma unroll
          for (int c = 0; c < HD; c += 32) {
            float v[32];
            tmem_ld32(ob + c, v);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[c + i] = o[c + i] * a_prev + v[i];
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&ofree[sp]);
        }
        a_prev = alpha;  // applied to O when O'_j is folded in at the next iteration
      } else {
        // after the last tile: fold O'_{n-1}
        const int sp = (j - 1) & 1;
        const uint32_t php = ((j - 1) >> 1) & 1;
        ok = mbar_wait(&ofull[sp], php, abort_flag, err, CORA_DERR_EPI_WAIT);
        if (!ok) break;
        tc_fence_after();
        const uint32_t ob = lane_base + 256 + sp * 128;
#pragma unroll
        for (int c = 0; c < HD; c += 32) {
          float v[32];
          tmem_ld32(ob + c, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[c + i] = o[c + i] * a_prev + v[i];
        }
        tc_fence_before();
      }
    }
    if (ok && q0 + r < S) {
      const float inv = 1.f / l;
      uint16_t* dst = out + static_cast<int64_t>(row_base + q0 + r) * (static_cast<int64_t>(Hq) * HD) + qcol;
#pragma unroll
      for (int c = 0; c < HD; c += 8) {
        *reinterpret_cast<uint4*>(dst + c) =
            make_uint4(pack_bf16x2(o[c] * inv, o[c + 1] * inv), pack_bf16x2(o[c + 2] * inv, o[c + 3] * inv),
                       pack_bf16x2(o[c + 4] * inv, o[c + 5] * inv), pack_bf16x2(o[c + 6] * inv, o[c + 7] * inv));
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

}  // namespace cora

using namespace cora;

cudaError_t attention_tc_prepare() {
  return cudaFuncSetAttribute(attention_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, attn::SMEM);
}

cudaError_t launch_attention_tc(const CUtensorMap& tmQKV, uint16_t* out, int B, int S, int Hq, int Hkv, int* err,
                                cudaStream_t st) {
  dim3 grid((S + attn::QT - 1) / attn::QT, Hq, B);
  return launch_pdl(attention_tc_kernel, grid, dim3(192), attn::SMEM, st, tmQKV, out, S, Hq, Hkv, err);
}
