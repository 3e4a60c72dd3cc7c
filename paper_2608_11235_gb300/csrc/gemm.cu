// Dense bf16 GEMM on the 5th-generation tensor cores (tcgen05) for the
// backbone's projections: acc[M, N] = A[M, K] * B[N, K]^T, fp32 accumulation
// in TMEM, operands staged in shared memory by TMA with 128-byte swizzling.
//
// Persistent stream-K kernel, one CTA per SM, 6 warps:
//   warp 0      TMA producer (one elected lane): A and B K-slices into a ring
//               of STAGES shared-memory buffers (full/empty mbarriers);
//   warp 1      TMEM allocator and MMA issuer (one lane): 128 x BN x 16
//               tcgen05.mma per K step, tcgen05.commit frees ring slots;
//   warps 2..5  epilogue: tcgen05.ld of the 128 x BN accumulator (warp w
//               reads TMEM lanes 32*(w%4) .. +31, one output row per thread),
//               fused epilogue, global stores.
//
// Work split (stream-K): the (tile, k-block) iterations of the whole GEMM
// are divided evenly among the CTAs, so every SM gets the same number of
// MMAs whatever the tile count.  A CTA's range is contiguous; only its first
// and last tile can be partial.  A tile split across CTAs is finished by the
// CTA that holds its k-block 0 (which reaches it at the END of its range);
// every other contributor writes its fp32 partial accumulator to its own
// workspace slot at the START of its range and raises a flag.  The finishing
// CTA adds the partials in increasing CTA order (deterministic), then runs the
// epilogue.  All CTAs are co-resident (grid <= SMs, one CTA per SM), waits are
// bounded, and the finishing CTA clears the flags it consumed.
//
// Tiles are ordered M-slowest, so at any moment the CTAs working on the same
// weight tile (B) for different row blocks run concurrently and share it
// through L2.  Two TMEM accumulators (2 * BN columns) let the epilogue of one
// segment overlap the MMAs of the next.
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

// Contiguous, even split of W iterations over G CTAs.
__device__ __forceinline__ int sk_start(int c, int G, int W) {
  return static_cast<int>((static_cast<long long>(c) * W) / G);
}

// A CTA's iteration range as segments (tile, kb0, kb1), visited in the order
// (1) its first segment (a contributor when it starts mid-tile), (2) its
// last segment (a split tile it finishes when it ends mid-tile), (3) the
// whole tiles in between.  Putting both split segments first lets their
// hand-off and fix-up overlap the MMAs of the whole tiles.
struct SegIter {
  int it0, it1, kb_per_tile, t_first, t_last, idx;
  __device__ SegIter(int c, int G, int W, int KB)
      : it0(sk_start(c, G, W)), it1(sk_start(c + 1, G, W)), kb_per_tile(KB), idx(0) {
    t_first = it0 / KB;
    t_last = it1 > it0 ? (it1 - 1) / KB : t_first - 1;
  }
  __device__ bool next(int& t, int& kb0, int& kb1) {
    if (it1 <= it0) return false;
    const int KB = kb_per_tile;
    if (t_first == t_last) {  // the whole range lies in one tile
      if (idx++ > 0) return false;
      t = t_first;
      kb0 = it0 - t * KB;
      kb1 = it1 - t * KB;
      return true;
    }
    const int n_mid = t_last - t_first - 1;
    if (idx >= 2 + n_mid) return false;
    if (idx == 0) {
      t = t_first;
      kb0 = it0 - t * KB;
      kb1 = KB;
    } else if (idx == 1) {
      t = t_last;
      kb0 = 0;
      kb1 = it1 - t * KB;
    } else {
      t = t_first + idx - 1;
      kb0 = 0;
      kb1 = KB;
    }
    ++idx;
    return true;
  }
};

__device__ __forceinline__ void red_add_v4(float* dst, const float* a) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(dst), "f"(a[0]), "f"(a[1]), "f"(a[2]), "f"(a[3])
               : "memory");
}

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

// Partial accumulators of split tiles: slot per CTA, [BN/16][128 rows][16]
// fp32, so a warp's 16-column chunk is 2 KB contiguous.
struct Partials {
  const float* slots[4];  // contributors' slots, in CTA order
  int n;
  int row;                // row within the tile (0..127)
};

__device__ __forceinline__ const float4* slot_chunk(const float* slot, int col, int row) {
  return reinterpret_cast<const float4*>(slot + (static_cast<int64_t>(col >> 4) * kBM + row) * 16);
}

// Loads four 16-column accumulator chunks (columns col[0..3]) under one TMEM
// wait, then adds every contributor's partial; all global loads of one
// contributor are issued before any is used, so the epilogue pays one memory
// round trip per four chunks instead of one per chunk.
__device__ __forceinline__ void load_acc64(uint32_t tacc, const int (&col)[4], const Partials& pp,
                                           float (&v)[4][16]) {
  uint32_t r[64];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%64];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, "
      "[%65];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47}, "
      "[%66];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, "
      "[%67];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
        "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
        "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
      : "r"(tacc + col[0]), "r"(tacc + col[1]), "r"(tacc + col[2]), "r"(tacc + col[3])
      : "memory");
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int i = 0; i < 16; ++i) v[q][i] = __uint_as_float(r[16 * q + i]);
  for (int p = 0; p < pp.n; ++p) {
    float4 x[4][4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4* src = slot_chunk(pp.slots[p], col[q], pp.row);
#pragma unroll
      for (int i = 0; i < 4; ++i) x[q][i] = __ldcg(src + i);
    }
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        v[q][4 * i] += x[q][i].x;
        v[q][4 * i + 1] += x[q][i].y;
        v[q][4 * i + 2] += x[q][i].z;
        v[q][4 * i + 3] += x[q][i].w;
      }
  }
}

// Epilogue of one 128 x BN tile for the calling thread's row, 64 columns
// (four chunks) per step.
template <int BN>
__device__ __forceinline__ void gemm_epilogue_row(const GemmEpilogue& ep, uint32_t tacc, int row, int M, int n0,
                                                  const Partials& pp) {
  const bool in_range = row < M;
  if (ep.mode == CORA_EPI_STORE_BF16) {
    uint16_t* crow = reinterpret_cast<uint16_t*>(ep.C) + static_cast<int64_t>(row) * ep.ldc + n0;
#pragma unroll 1
    for (int c = 0; c < BN; c += 64) {
      float v[4][16];
      const int cols[4] = {c, c + 16, c + 32, c + 48};
      load_acc64(tacc, cols, pp, v);
      if (in_range)
#pragma unroll
        for (int q = 0; q < 4; ++q) store_bf16x16(crow + c + 16 * q, v[q]);
    }
  } else if (ep.mode == CORA_EPI_RESID_F32) {
    // h += acc as vector reductions performed at L2: no read round trip, and
    // exactly one add per element per launch, so the result is deterministic.
    float* crow = reinterpret_cast<float*>(ep.C) + static_cast<int64_t>(row) * ep.ldc + n0;
#pragma unroll 1
    for (int c = 0; c < BN; c += 64) {
      float v[4][16];
      const int cols[4] = {c, c + 16, c + 32, c + 48};
      load_acc64(tacc, cols, pp, v);
      if (in_range)
#pragma unroll
        for (int i = 0; i < 16; ++i) red_add_v4(crow + c + 4 * i, &v[i >> 2][(i & 3) * 4]);
    }
  } else if (ep.mode == CORA_EPI_SWIGLU) {
    // Tile columns [0, BN/2) are gate rows, [BN/2, BN) the matching up rows
    // of output features n0/2 .. n0/2 + BN/2.
    uint16_t* crow = reinterpret_cast<uint16_t*>(ep.C) + static_cast<int64_t>(row) * ep.ldc + n0 / 2;
#pragma unroll 1
    for (int c = 0; c < BN / 2; c += 32) {
      float v[4][16];
      const int cols[4] = {c, c + 16, BN / 2 + c, BN / 2 + c + 16};
      load_acc64(tacc, cols, pp, v);
#pragma unroll
      for (int q = 0; q < 2; ++q)
#pragma unroll
        for (int j = 0; j < 16; ++j) v[q][j] = silu_f(v[q][j]) * v[q + 2][j];
      if (in_range) {
        store_bf16x16(crow + c, v[0]);
        store_bf16x16(crow + c + 16, v[1]);
      }
    }
  } else {  // CORA_EPI_ROPE_BF16: rotate pairs (j, j + hd/2) of every head
    uint16_t* crow = reinterpret_cast<uint16_t*>(ep.C) + static_cast<int64_t>(row) * ep.ldc + n0;
    const int hd = ep.head_dim, half = hd / 2;
    const int pos = in_range ? row % ep.seq : 0;
    const float2* tab = reinterpret_cast<const float2*>(ep.rope) + static_cast<int64_t>(pos) * half;
#pragma unroll 1
    for (int h0 = 0; h0 < BN; h0 += hd) {
      const bool rot = n0 + h0 < ep.rope_cols;
#pragma unroll 1
      for (int j0 = 0; j0 < half; j0 += 32) {
        float v[4][16];
        const int cols[4] = {h0 + j0, h0 + j0 + 16, h0 + half + j0, h0 + half + j0 + 16};
        load_acc64(tacc, cols, pp, v);
        if (rot) {
#pragma unroll
          for (int q = 0; q < 2; ++q)
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float2 cs = tab[j0 + 16 * q + j];
              const float a = v[q][j], b = v[q + 2][j];
              v[q][j] = a * cs.x - b * cs.y;
              v[q + 2][j] = b * cs.x + a * cs.y;
            }
        }
        if (in_range) {
          store_bf16x16(crow + h0 + j0, v[0]);
          store_bf16x16(crow + h0 + j0 + 16, v[1]);
          store_bf16x16(crow + h0 + half + j0, v[2]);
          store_bf16x16(crow + h0 + half + j0 + 16, v[3]);
        }
      }
    }
  }
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.global.acquire.gpu.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Bounded spin until *flag != 0.
__device__ __forceinline__ bool wait_flag(const int* flag, volatile int* abort, int* err) {
  const long long t0 = clock64();
  while (ld_acquire(flag) == 0) {
    if (*abort) return false;
    if (clock64() - t0 > CORA_WAIT_LIMIT) {
      record_error(err, CORA_DERR_SPLIT_WAIT);
      *abort = 1;
      return false;
    }
    __nanosleep(100);
  }
  return true;
}

template <int BN>
__global__ void __launch_bounds__(192, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, int M, int N,
                   int K, GemmEpilogue ep, GemmWorkspace ws, int* err) {
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
  const int num_n = N / BN;
  const int num_tiles = ((M + kBM - 1) / kBM) * num_n;
  const int KB = K / kBK;
  const int W = num_tiles * KB;
  const int G = gridDim.x;

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
      SegIter seg(blockIdx.x, G, W, KB);
      int t, kb0, kb1;
      while (seg.next(t, kb0, kb1)) {
        const int mb = t / num_n, nb = t - mb * num_n;
        for (int kb = kb0; kb < kb1; ++kb) {
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
      SegIter seg(blockIdx.x, G, W, KB);
      int t, kb0, kb1;
      while (seg.next(t, kb0, kb1)) {
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        ++it;
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, err, CORA_DERR_MMA_WAIT)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
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
                      (kb > kb0 || k > 0) ? 1u : 0u);
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
    const int etid = threadIdx.x - 64;
    const int row_local = sub * 32 + lane;
    int it = 0;
    SegIter seg(blockIdx.x, G, W, KB);
    int t, kb0, kb1;
    while (seg.next(t, kb0, kb1)) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      ++it;
      const bool ok = mbar_wait(&tfull[acc], acc_phase, abort_flag, err, CORA_DERR_EPI_WAIT);
      if (named_bar_or(1, 128, !ok)) break;  // uniform exit of the four epilogue warps
      tc_fence_after();
      const int mb = t / num_n, nb = t - mb * num_n;
      const uint32_t tacc = tmem_base + (static_cast<uint32_t>(sub * 32) << 16) + acc * BN;
      if (kb0 > 0) {
        // Contributor: hand the partial accumulator to the tile's finisher.
        float* slot = ws.partial + static_cast<int64_t>(blockIdx.x) * kBM * BN;
        Partials none;
        none.n = 0;
        none.row = row_local;
#pragma unroll 1
        for (int c = 0; c < BN; c += 64) {
          float v[4][16];
          const int cols[4] = {c, c + 16, c + 32, c + 48};
          load_acc64(tacc, cols, none, v);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float4* dst = reinterpret_cast<float4*>(slot + (static_cast<int64_t>((c >> 4) + q) * kBM + row_local) * 16);
#pragma unroll
            for (int i = 0; i < 4; ++i)
              dst[i] = make_float4(v[q][4 * i], v[q][4 * i + 1], v[q][4 * i + 2], v[q][4 * i + 3]);
          }
        }
        tc_fence_before();
        mbar_arrive(&tempty[acc]);
        __threadfence();
        named_bar_sync(1, 128);
        if (etid == 0) atomicExch(ws.flags + blockIdx.x, 1);
        continue;
      }
      Partials pp;
      pp.n = 0;
      pp.row = row_local;
      int c_first = 0, c_last = -1;
      if (kb1 < KB) {
        // Finisher of a split tile: contributors are the next CTAs up to the
        // one whose range holds the tile's last k-block.
        const int last_it = t * KB + KB - 1;
        c_first = blockIdx.x + 1;
        c_last = c_first;
        while (c_last + 1 < G && sk_start(c_last + 1, G, W) <= last_it) ++c_last;
        bool fok = true;
        if (etid == 0)
          for (int c = c_first; c <= c_last && fok; ++c) fok = wait_flag(ws.flags + c, abort_flag, err);
        if (named_bar_or(1, 128, !fok)) break;
        for (int c = c_first; c <= c_last; ++c) {
          (void)ld_acquire(ws.flags + c);
          if (pp.n < 4) pp.slots[pp.n++] = ws.partial + static_cast<int64_t>(c) * kBM * BN;
        }
        if (c_last - c_first + 1 > 4) record_error(err, CORA_DERR_SPLIT_WAIT);  // cannot happen: grid checked
      }
      gemm_epilogue_row<BN>(ep, tacc, mb * kBM + row_local, M, nb * BN, pp);
      tc_fence_before();
      mbar_arrive(&tempty[acc]);
      if (c_last >= c_first) {
        named_bar_sync(1, 128);  // every thread has read the partials
        if (etid == 0)
          for (int c = c_first; c <= c_last; ++c) atomicExch(ws.flags + c, 0);
      }
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

size_t gemm_workspace_bytes(int num_sms) { return static_cast<size_t>(num_sms) * kBM * 256 * sizeof(float); }

// Grid for a stream-K launch: one CTA per SM, but every CTA gets at least
// ceil(KB/4) iterations, so a split tile has at most four contributors
// besides its finisher; never more CTAs than iterations.
static int gemm_grid(int M, int N, int K, int bn, int num_sms) {
  const int tiles = ((M + kBM - 1) / kBM) * (N / bn);
  const int KB = K / kBK;
  const long long W = static_cast<long long>(tiles) * KB;
  long long g = num_sms;
  const long long max_by_share = W / ((KB + 3) / 4);
  if (g > max_by_share) g = max_by_share;
  if (g > W) g = W;
  return g < 1 ? 1 : static_cast<int>(g);
}

template <int BN>
static cudaError_t launch_gemm_bn(const CUtensorMap& tmA, const CUtensorMap& tmB, int M, int N, int K,
                                  const GemmEpilogue& ep, const GemmWorkspace& ws, int* err, int num_sms,
                                  cudaStream_t st) {
  using Cfg = GemmCfg<BN>;
  const int grid = gemm_grid(M, N, K, BN, num_sms);
  gemm_tc_kernel<BN><<<grid, 192, Cfg::SMEM_BYTES, st>>>(tmA, tmB, M, N, K, ep, ws, err);
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
                        const GemmWorkspace& ws, int* err, int num_sms, cudaStream_t st) {
  if (gemm_block_n(N, ep.mode) == 256) return launch_gemm_bn<256>(tmA, tmB, M, N, K, ep, ws, err, num_sms, st);
  return launch_gemm_bn<128>(tmA, tmB, M, N, K, ep, ws, err, num_sms, st);
}
