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
//
// Many tiles (the 2-CTA kernel, more than two row blocks, at least one tile
// per unit): stream-K covers only the remainder, tiles mod units, and the
// rest run as whole tiles in data-parallel waves (unit c takes tile
// sk + w P + c in wave w), with tiles numbered in groups of row blocks, row
// block fastest (see tile_coords).  A contiguous range per unit over
// thousands of tiles would put the units' concurrent tiles all over the tile
// grid, every one on its own weight tile, each unit at its own k-offset; a
// wave of consecutive tiles covers a few row blocks and weight tiles, every
// unit at the same k-block, so each k-slice of a shared operand comes from
// DRAM once and from L2 for the other units.
#include <math.h>

#include <algorithm>

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
  // Epilogue staging: 4 warps x 2 buffers x (32 rows x 128 bytes), 128-byte
  // swizzled, the source of the TMA stores / reductions of the outputs.
  static constexpr int STG_BYTES = 4 * 2 * 4096;
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + STG_BYTES + 1024 /*align*/ + 256 /*barriers*/;
};

// Division of the W = tiles * KB (tile, k-block) iterations among G CTAs
// (or CTA pairs).  Uniform (stream-K): unit c starts at c W / G.  Skewed
// equal splits (G = tiles * S): the piece holding k-block 0, which finishes
// the tile, is skew * (S - 1) k-blocks longer than KB / S and every other
// piece skew shorter, so the other pieces' partials are written while the
// finisher is still issuing MMAs instead of after.
struct WorkSplit {
  int G, W, KB, S, skew;  // G: the units sharing the stream-K tiles (the first W / KB)
  // Whole tiles each of the P units runs after its stream-K range: unit c
  // runs tile W / KB + w P + c in wave w.
  int dp_waves, P;
  __host__ __device__ int start(int c) const {
    if (skew > 0) {
      const int t = c / S, s = c - t * S;
      return t * KB + (s == 0 ? 0 : KB - (S - s) * (KB / S - skew));
    }
    return static_cast<int>((static_cast<long long>(c) * W) / G);
  }
};

// A CTA's iteration range as segments (tile, kb0, kb1), visited in the order
// (1) its first segment (a contributor when it starts mid-tile), (2) its
// last segment (a split tile it finishes when it ends mid-tile), (3) the
// whole tiles in between, (4) its data-parallel tiles.  Putting both split
// segments first lets their hand-off and fix-up overlap the MMAs of the
// whole tiles.
struct SegIter {
  int it0, it1, kb_per_tile, t_first, t_last, idx, n_sk, dp_t0, dp_stride, dp_n;
  __host__ __device__ SegIter(int c, const WorkSplit& ws)
      : it0(c < ws.G ? ws.start(c) : ws.W), it1(c < ws.G ? ws.start(c + 1) : ws.W), kb_per_tile(ws.KB), idx(0) {
    t_first = it0 / ws.KB;
    t_last = it1 > it0 ? (it1 - 1) / ws.KB : t_first - 1;
    n_sk = it1 <= it0 ? 0 : (t_first == t_last ? 1 : 2 + (t_last - t_first - 1));
    dp_t0 = ws.W / ws.KB + c;
    dp_stride = ws.P;
    dp_n = ws.dp_waves;
  }
  __host__ __device__ bool next(int& t, int& kb0, int& kb1) {
    const int KB = kb_per_tile;
    if (idx >= n_sk) {  // data-parallel whole tiles
      const int w = idx - n_sk;
      if (w >= dp_n) return false;
      t = dp_t0 + w * dp_stride;
      kb0 = 0;
      kb1 = KB;
      ++idx;
      return true;
    }
    if (t_first == t_last) {  // the whole stream-K range lies in one tile
      t = t_first;
      kb0 = it0 - t * KB;
      kb1 = it1 - t * KB;
    } else if (idx == 0) {
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
  // True once the segment just returned is the last one this CTA visits.
  __host__ __device__ bool finished() const { return idx >= n_sk + dp_n; }
};

// Row block and column block of tile t: tiles are numbered in groups of
// `group` row blocks (the last group may be smaller), row block fastest
// within a group, so consecutive tiles share weight tiles (B) and the group's
// row blocks (A) stay in L2 while its columns are walked.  group = 1: M-slowest.
__host__ __device__ __forceinline__ void tile_coords(int t, int num_m, int num_n, int group, int& mb, int& nb) {
  const int per_group = group * num_n;
  const int g = t / per_group, r = t - g * per_group;
  const int gm = min(group, num_m - g * group);
  mb = g * group + r % gm;
  nb = r / gm;
}

// Walks a CTA's (tile, k-block) sequence in the order the producer loads it.
struct KbCursor {
  SegIter seg;
  int t, kb, kb1;
  bool valid;
  __device__ KbCursor(int c, const WorkSplit& ws) : seg(c, ws) {
    int kb0 = 0;
    valid = seg.next(t, kb0, kb1);
    kb = kb0;
  }
  __device__ void advance() {
    if (!valid) return;
    if (++kb >= kb1) {
      int kb0 = 0;
      valid = seg.next(t, kb0, kb1);
      kb = kb0;
    }
  }
};

__device__ __forceinline__ void red_add_v4(float* dst, const float* a) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(dst), "f"(a[0]), "f"(a[1]), "f"(a[2]), "f"(a[3])
               : "memory");
}

// silu(x) = x / (1 + e^-x); the approximate divide is within 2 ulp (the
// result is rounded to bf16), and for x -> -inf the denominator overflows to
// inf and the quotient goes to -0 as the exact function does.
__device__ __forceinline__ float silu_f(float x) { return __fdividef(x, 1.f + __expf(-x)); }

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

// Partial accumulators of split tiles: slot per CTA, [BN/16][4][128 rows][4]
// fp32.  Thread r owns row r; its float4 i of 16-column chunk q sits at
// index (4 q + i) * 128 + r, so one warp-wide float4 access covers 512
// contiguous bytes (whole 128-byte lines in global memory, no bank conflicts
// in shared memory).
struct Partials {
  const float* slots[4];  // contributors' slots, in CTA order
  int n;
  int row;                // row within the tile (0..127)
  bool in_smem;           // slots were bulk-copied into this CTA's shared memory
};

__device__ __forceinline__ int part_f4(int col, int i, int row) { return ((col >> 4) * 4 + i) * kBM + row; }

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
      const float4* src = reinterpret_cast<const float4*>(pp.slots[p]);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int o = part_f4(col[q], i, pp.row);
        x[q][i] = pp.in_smem ? src[o] : __ldcg(src + o);
      }
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

// ------------------------------------------------------------ TMA epilogue
// Each epilogue warp owns rows [32*sub, 32*sub + 32) of the tile and two
// 4 KB staging buffers.  A "unit" is 32 rows x 128 bytes (64 bf16 or 32 fp32
// columns): every thread writes its row into the buffer with the 128-byte
// swizzle (16-byte chunk j of row r at chunk j ^ (r % 8): conflict-free), and
// lane 0 hands the unit to TMA as one 2-D store (bf16 outputs) or one 2-D
// fp32 reduce-add (the residual stream), i.e. whole 128-byte lines.
struct Stager {
  uint8_t* buf[2];
  int cur;
  int lane;
};

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* src, int c0, int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1)
               : "memory");
}

__device__ __forceinline__ void tma_reduce_add_2d(const CUtensorMap* map, const void* src, int c0, int c1) {
  asm volatile("cp.reduce.async.bulk.tensor.2d.global.shared::cta.add.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1)
               : "memory");
}

__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }

template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}


// Next staging buffer, once the TMA operation that last read it is done.
__device__ __forceinline__ uint8_t* stage_acquire(Stager& sg) {
  sg.cur ^= 1;
  if (sg.lane == 0) bulk_wait_read<1>();
  __syncwarp();
  return sg.buf[sg.cur];
}

// Write 16 bytes (chunk j of this thread's row) into a swizzled unit.
__device__ __forceinline__ void stage_chunk(uint8_t* unit, int lane, int j, uint4 v) {
  *reinterpret_cast<uint4*>(unit + lane * 128 + ((j ^ (lane & 7)) << 4)) = v;
}

__device__ __forceinline__ void stage_bf16x16(uint8_t* unit, int lane, int j0, const float (&v)[16]) {
  stage_chunk(unit, lane, j0, make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                         pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7])));
  stage_chunk(unit, lane, j0 + 1, make_uint4(pack_bf16x2(v[8], v[9]), pack_bf16x2(v[10], v[11]),
                                             pack_bf16x2(v[12], v[13]), pack_bf16x2(v[14], v[15])));
}

__device__ __forceinline__ void stage_f32x16(uint8_t* unit, int lane, int j0, const float (&v)[16]) {
#pragma unroll
  for (int q = 0; q < 4; ++q)
    stage_chunk(unit, lane, j0 + q,
                make_uint4(__float_as_uint(v[4 * q]), __float_as_uint(v[4 * q + 1]), __float_as_uint(v[4 * q + 2]),
                           __float_as_uint(v[4 * q + 3])));
}

__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, const void* src, int c0, int c1, int c2) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1), "r"(c2)
               : "memory");
}

// Make the warp's staged unit visible to the async proxy and issue it
// (c2 >= 0: a 3-D store at {c0, c1, c2}).
__device__ __forceinline__ void stage_issue(const Stager& sg, const CUtensorMap* map, const uint8_t* unit, int c0,
                                            int c1, bool reduce, int c2 = -1) {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  __syncwarp();
  if (sg.lane == 0) {
    if (reduce)
      tma_reduce_add_2d(map, unit, c0, c1);
    else if (c2 >= 0)
      tma_store_3d(map, unit, c0, c1, c2);
    else
      tma_store_2d(map, unit, c0, c1);
    bulk_commit();
  }
}

// Epilogue of one 128 x BN tile for this warp's 32 rows (row0 = first global
// row of the warp's box).  STORE and RESID write tile columns [c_lo, c_hi)
// only (multiples of 64); the other modes always write the whole tile.
template <int BN>
__device__ __forceinline__ void gemm_epilogue_warp(const GemmEpilogue& ep, const CUtensorMap* tmC, uint32_t tacc,
                                                   int row0, int n0, const Partials& pp, Stager& sg, int c_lo = 0,
                                                   int c_hi = BN) {
  const int lane = sg.lane;
  if (ep.mode == CORA_EPI_STORE_BF16) {
#pragma unroll 1
    for (int c = c_lo; c < c_hi; c += 64) {
      float v[4][16];
      const int cols[4] = {c, c + 16, c + 32, c + 48};
      load_acc64(tacc, cols, pp, v);
      uint8_t* u = stage_acquire(sg);
#pragma unroll
      for (int q = 0; q < 4; ++q) stage_bf16x16(u, lane, 2 * q, v[q]);
      stage_issue(sg, tmC, u, n0 + c, row0, false);
    }
  } else if (ep.mode == CORA_EPI_RESID_F32) {
#pragma unroll 1
    for (int c = c_lo; c < c_hi; c += 64) {
      float v[4][16];
      const int cols[4] = {c, c + 16, c + 32, c + 48};
      load_acc64(tacc, cols, pp, v);
      if (lane == 0) bulk_wait_read<0>();  // both buffers free
      __syncwarp();
      stage_f32x16(sg.buf[0], lane, 0, v[0]);
      stage_f32x16(sg.buf[0], lane, 4, v[1]);
      stage_f32x16(sg.buf[1], lane, 0, v[2]);
      stage_f32x16(sg.buf[1], lane, 4, v[3]);
      stage_issue(sg, tmC, sg.buf[0], n0 + c, row0, true);
      stage_issue(sg, tmC, sg.buf[1], n0 + c + 32, row0, true);
      sg.cur = 1;
    }
  } else if (ep.mode == CORA_EPI_SWIGLU) {
    // Tile columns [0, BN/2) are gate rows, [BN/2, BN) the matching up rows of
    // output features n0/2 .. n0/2 + BN/2.
#pragma unroll 1
    for (int c = 0; c < BN / 2; c += 64) {
      uint8_t* u = stage_acquire(sg);
#pragma unroll 1
      for (int h = 0; h < 64; h += 32) {
        float v[4][16];
        const int cols[4] = {c + h, c + h + 16, BN / 2 + c + h, BN / 2 + c + h + 16};
        load_acc64(tacc, cols, pp, v);
#pragma unroll
        for (int q = 0; q < 2; ++q) {
#pragma unroll
          for (int j = 0; j < 16; ++j) v[q][j] = silu_f(v[q][j]) * v[q + 2][j];
          stage_bf16x16(u, lane, (h >> 3) + 2 * q, v[q]);
        }
      }
      stage_issue(sg, tmC, u, n0 / 2 + c, row0, false);
    }
  } else {  // CORA_EPI_ROPE_BF16: rotate pairs (j, j + hd/2) of every head
    const int hd = ep.head_dim, half = hd / 2;
    const int pos = ep.rope_pos0 + (row0 + lane >= 0 ? (row0 + lane) % ep.seq : 0);
    // store coordinates of the warp's 32-row box (they never straddle a sequence: seq % 32 == 0 when out3d)
    const int srow = ep.out3d ? ep.rope_pos0 + row0 % ep.seq : row0, sseq = ep.out3d ? row0 / ep.seq : -1;
    const float2* tab = reinterpret_cast<const float2*>(ep.rope_t) + pos;  // frequency j at tab[j * rope_tn]
#pragma unroll 1
    for (int h0 = 0; h0 < BN; h0 += hd) {
      const bool rot = n0 + h0 < ep.rope_cols;
      // hd = 128: the two halves go to two units (both buffers); hd = 64: one unit.
      uint8_t* u1;
      uint8_t* u2;
      if (hd == 128) {
        if (lane == 0) bulk_wait_read<0>();
        __syncwarp();
        u1 = sg.buf[0];
        u2 = sg.buf[1];
        sg.cur = 1;
      } else {
        u1 = stage_acquire(sg);
        u2 = u1;
      }
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
              const float2 cs = tab[static_cast<int64_t>(j0 + 16 * q + j) * ep.rope_tn];
              const float a = v[q][j], b = v[q + 2][j];
              v[q][j] = a * cs.x - b * cs.y;
              v[q + 2][j] = b * cs.x + a * cs.y;
            }
        }
        // chunk index (16 bytes = 8 bf16) of column x within a 64-column unit
        const int k1 = j0 >> 3;
        const int k2 = hd == 128 ? (j0 >> 3) : ((half + j0) >> 3);
        stage_bf16x16(u1, lane, k1, v[0]);
        stage_bf16x16(u1, lane, k1 + 2, v[1]);
        stage_bf16x16(u2, lane, k2, v[2]);
        stage_bf16x16(u2, lane, k2 + 2, v[3]);
      }
      if (hd == 128) {
        stage_issue(sg, tmC, u1, n0 + h0, srow, false, sseq);
        stage_issue(sg, tmC, u2, n0 + h0 + half, srow, false, sseq);
      } else {
        stage_issue(sg, tmC, u1, n0 + h0, srow, false, sseq);
      }
    }
  }
}

// Contiguous global -> shared bulk copy completing `bytes` on `bar`.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
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

// Paired fix-up of a tile split into two k-pieces: each piece finalises half
// of the tile's columns.  This writes the accumulator columns
// [give_lo, give_lo + BN/2) that the other piece finalises into this piece's
// slot, raises this piece's flag and waits for the other's, so the caller can
// add the other piece's slot over its own half.  Both pieces are resident
// (one CTA per SM, grid <= SMs) and the wait is bounded.  With two terms the
// sum is the same whichever piece adds it, so results stay deterministic.
template <int BN>
__device__ __forceinline__ bool pair_exchange(uint32_t tacc, int give_lo, float* my_slot, int* my_flag,
                                              const int* other_flag, int row_local, int etid,
                                              volatile int* abort_flag, int* err) {
  Partials none;
  none.n = 0;
  none.row = row_local;
  none.in_smem = false;
#pragma unroll 1
  for (int c = give_lo; c < give_lo + BN / 2; c += 64) {
    float v[4][16];
    const int cols[4] = {c, c + 16, c + 32, c + 48};
    load_acc64(tacc, cols, none, v);
    float4* dst = reinterpret_cast<float4*>(my_slot);
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
      for (int i = 0; i < 4; ++i)
        dst[part_f4(c + 16 * q, i, row_local)] =
            make_float4(v[q][4 * i], v[q][4 * i + 1], v[q][4 * i + 2], v[q][4 * i + 3]);
  }
  __threadfence();
  named_bar_sync(1, 128);
  bool fok = true;
  if (etid == 0) {
    atomicExch(my_flag, 1);
    fok = wait_flag(other_flag, abort_flag, err);
  }
  if (named_bar_or(1, 128, !fok)) return false;
  (void)ld_acquire(other_flag);
  return true;
}

template <int BN>
__global__ void __launch_bounds__(192, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, int M, int N, int K, GemmEpilogue ep, GemmWorkspace ws,
                   int* err) {
  using Cfg = GemmCfg<BN>;
  constexpr int STAGES = Cfg::STAGES;
  constexpr uint32_t IDESC = idesc_bf16_f32(kBM, BN);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* stg = smem + STAGES * Cfg::STAGE_BYTES;  // epilogue staging (1024-aligned)
  uint64_t* full = reinterpret_cast<uint64_t*>(stg + Cfg::STG_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* pbar = tempty + 2;  // completion of bulk partial copies
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(pbar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t pbar_phase = 0;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_n = N / BN;
  const int num_tiles = ((M + kBM - 1) / kBM) * num_n;
  const int KB = K / kBK;
  const int W = num_tiles * KB;
  const int G = gridDim.x;
  const WorkSplit wsplit{G, W, KB, ep.splits, ep.split_skew, 0, G};

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 128);
    }
    mbar_init(pbar, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    tma_prefetch_desc(&tmC);
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
  pdl_wait();  // A, the outputs and the workspace belong to the previous kernels

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      SegIter seg(blockIdx.x, wsplit);
      int t, kb0, kb1;
      while (seg.next(t, kb0, kb1)) {
        const int mb = t / num_n, nb = t - mb * num_n;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err, CORA_DERR_TMA_WAIT)) goto producer_done;
          uint8_t* sa = smem + stage * Cfg::STAGE_BYTES;
          mbar_arrive_expect_tx(&full[stage], Cfg::STAGE_BYTES);
          tma_load_2d(sa, &tmA, &full[stage], kb * kBK, mb * kBM);
          // B boxes are 128 rows (the same maps feed the 2-CTA kernel's halves).
#pragma unroll
          for (int h = 0; h < BN / 128; ++h)
            tma_load_2d(sa + Cfg::A_BYTES + h * 16384, &tmB, &full[stage], kb * kBK, nb * BN + h * 128);
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
      SegIter seg(blockIdx.x, wsplit);
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
    Stager sg;
    sg.buf[0] = stg + sub * 8192;
    sg.buf[1] = stg + sub * 8192 + 4096;
    sg.cur = 1;
    sg.lane = lane;
    int it = 0;
    SegIter seg(blockIdx.x, wsplit);
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
      if (ep.split_pair) {
        // Two k-pieces per tile (CTA 2t + s): piece s finalises columns
        // [s BN/2, (s+1) BN/2).
        const int me = blockIdx.x, other = blockIdx.x ^ 1, s = blockIdx.x & 1;
        if (!pair_exchange<BN>(tacc, (1 - s) * (BN / 2), ws.partial + static_cast<int64_t>(me) * kBM * BN,
                               ws.flags + me, ws.flags + other, row_local, etid, abort_flag, err))
          break;
        Partials pp;
        pp.n = 1;
        pp.row = row_local;
        pp.in_smem = false;
        pp.slots[0] = ws.partial + static_cast<int64_t>(other) * kBM * BN;
        gemm_epilogue_warp<BN>(ep, &tmC, tacc, mb * kBM + sub * 32, nb * BN, pp, sg, s * (BN / 2), (s + 1) * (BN / 2));
        tc_fence_before();
        mbar_arrive(&tempty[acc]);
        named_bar_sync(1, 128);  // every thread has read the other piece's slot
        if (etid == 0) atomicExch(ws.flags + other, 0);
        continue;
      }
      if (kb0 > 0) {
        // Contributor: hand the partial accumulator to the tile's finisher.
        float* slot = ws.partial + static_cast<int64_t>(blockIdx.x) * kBM * BN;
        Partials none;
        none.n = 0;
        none.row = row_local;
        none.in_smem = false;
#pragma unroll 1
        for (int c = 0; c < BN; c += 64) {
          float v[4][16];
          const int cols[4] = {c, c + 16, c + 32, c + 48};
          load_acc64(tacc, cols, none, v);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float4* dst = reinterpret_cast<float4*>(slot);
#pragma unroll
            for (int i = 0; i < 4; ++i)
              dst[part_f4(c + 16 * q, i, row_local)] =
                  make_float4(v[q][4 * i], v[q][4 * i + 1], v[q][4 * i + 2], v[q][4 * i + 3]);
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
      pp.in_smem = false;
      int c_first = 0, c_last = -1;
      if (kb1 < KB) {
        // Finisher of a split tile: contributors are the next CTAs up to the
        // one whose range holds the tile's last k-block.
        const int last_it = t * KB + KB - 1;
        c_first = blockIdx.x + 1;
        c_last = c_first;
        while (c_last + 1 < G && wsplit.start(c_last + 1) <= last_it) ++c_last;
        const int n_c = c_last - c_first + 1;
        // When no segment follows, the operand ring is idle (every MMA of this
        // CTA has completed): bulk-copy the contributors' partials into it.
        const bool bulk = seg.finished() && n_c * kBM * BN * 4 <= STAGES * Cfg::STAGE_BYTES;
        bool fok = true;
        if (etid == 0) {
          for (int c = c_first; c <= c_last && fok; ++c) fok = wait_flag(ws.flags + c, abort_flag, err);
          if (fok && bulk) {
            asm volatile("fence.proxy.async.global;" ::: "memory");
            const uint32_t bytes = kBM * BN * 4;
            mbar_arrive_expect_tx(pbar, bytes * n_c);
            for (int c = c_first; c <= c_last; ++c)
              bulk_g2s(smem + (c - c_first) * bytes, ws.partial + static_cast<int64_t>(c) * kBM * BN, bytes, pbar);
          }
        }
        if (named_bar_or(1, 128, !fok)) break;
        if (bulk) {
          const bool bok = mbar_wait(pbar, pbar_phase, abort_flag, err, CORA_DERR_SPLIT_WAIT);
          pbar_phase ^= 1u;
          if (named_bar_or(1, 128, !bok)) break;
          pp.in_smem = true;
          for (int c = c_first; c <= c_last && pp.n < 4; ++c)
            pp.slots[pp.n++] = reinterpret_cast<const float*>(smem) + static_cast<int64_t>(c - c_first) * kBM * BN;
        } else {
          for (int c = c_first; c <= c_last; ++c) {
            (void)ld_acquire(ws.flags + c);
            if (pp.n < 4) pp.slots[pp.n++] = ws.partial + static_cast<int64_t>(c) * kBM * BN;
          }
        }
        if (n_c > 4) record_error(err, CORA_DERR_SPLIT_WAIT);  // cannot happen: grid rule
      }
      gemm_epilogue_warp<BN>(ep, &tmC, tacc, mb * kBM + sub * 32, nb * BN, pp, sg);
      tc_fence_before();
      mbar_arrive(&tempty[acc]);
      if (c_last >= c_first) {
        named_bar_sync(1, 128);  // every thread has read the partials
        if (etid == 0)
          for (int c = c_first; c <= c_last; ++c) atomicExch(ws.flags + c, 0);
      }
    }
    // The staging buffers must be read out before the CTA retires; the
    // global writes themselves complete with the grid (and are visible to a
    // dependent grid after its griddepcontrol.wait).
    if (lane == 0) bulk_wait_read<0>();
    __syncwarp();
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

// ======================================================================
// 2-CTA variant (cta_group::2): a cluster of two CTAs on two SMs computes a
// 256 x 256 tile.  Each CTA stages its own 128 rows of A and its own 128-row
// half of B per K step (32 KB per stage, 6 stages), so each SM moves half as
// many operand bytes per MMA as the 1-CTA kernel; the even CTA issues
// tcgen05.mma.cta_group::2 (M = 256, N = 256), whose result lands in both
// CTAs' TMEM (each its own 128 rows).  Both CTAs' TMA loads complete on the
// leader's full barrier; the leader's commits are multicast to both CTAs'
// empty / accumulator-ready barriers; both CTAs' epilogue warps release the
// leader's accumulator barrier.  Work split and epilogues are those of the
// 1-CTA kernel, applied to pair-tiles (a pair is one stream-K unit; CTA
// 2p + r owns partial slot / flag 2p + r for its 128 rows).
// ======================================================================
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map, uint32_t bar_cluster, int c0,
                                                 int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cta.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, {%3, "
      "%4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(c0), "r"(c1)
      : "memory");
}

__device__ __forceinline__ void umma2_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on the barrier at this offset in both CTAs of the pair when the
// leader's MMAs issued so far are done.
__device__ __forceinline__ void umma2_commit_both(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          smem_u32(bar)),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}

__device__ __forceinline__ void mbar_arrive_remote(uint32_t bar_cluster) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}

struct Gemm2Cfg {
  static constexpr int A_BYTES = kBM * kBK * 2;      // this CTA's 128 rows of A
  static constexpr int B_BYTES = 128 * kBK * 2;      // this CTA's half of B
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = 6;
  static constexpr int TMEM_COLS = 512;              // two 256-column accumulators
  static constexpr int STG_BYTES = 4 * 2 * 4096;
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + STG_BYTES + 1024 + 256;
};

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(192, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmC, int M, int N, int K, GemmEpilogue ep, GemmWorkspace ws,
                    int* err) {
  using Cfg = Gemm2Cfg;
  constexpr int BN = 256;
  constexpr int STAGES = Cfg::STAGES;
  constexpr uint32_t IDESC = idesc_bf16_f32(256, BN);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* stg = smem + STAGES * Cfg::STAGE_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(stg + Cfg::STG_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* pbar = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(pbar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t pbar_phase = 0;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int pair = blockIdx.x >> 1;
  const int G = gridDim.x >> 1;
  const int num_n = N / BN;
  const int num_m = (M + 255) / 256;
  const int num_tiles = num_m * num_n;
  const int KB = K / kBK;
  const int W = (num_tiles - ep.dp_waves * G) * KB;  // the stream-K tiles' iterations
  const WorkSplit wsplit{ep.sk_units, W, KB, ep.splits, ep.split_skew, ep.dp_waves, G};
  const int group = ep.raster_group;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 8);  // one arrival per epilogue warp of both CTAs
    }
    mbar_init(pbar, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    tma_prefetch_desc(&tmC);
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(Cfg::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  __syncwarp();  // converged arrival (one lane of warp 0 initialised the barriers)
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers initialised before any cross-CTA signal
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_trigger();

  // With ep.b_static, the ring's first B tiles are loaded before waiting for
  // the previous kernel: B (the weights) does not depend on it, A does.
  const int b_row = static_cast<int>(rank) * 128;
  int n_pre = 0, n_issued = 0;
  if (warp == 0 && lane == 0 && ep.b_static) {
    for (KbCursor cur(pair, wsplit); n_pre < STAGES && cur.valid; ++n_pre, cur.advance()) {
      uint8_t* sa = smem + n_pre * Cfg::STAGE_BYTES;
      if (leader) mbar_arrive_expect_tx(&full[n_pre], 2 * Cfg::STAGE_BYTES);
      int pmb, pnb;
      tile_coords(cur.t, num_m, num_n, group, pmb, pnb);
      tma_load_2d_pair(sa + Cfg::A_BYTES, &tmB, mapa_shared(smem_u32(&full[n_pre]), 0), cur.kb * kBK,
                       pnb * BN + b_row);
    }
  }
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      SegIter seg(pair, wsplit);
      int t, kb0, kb1;
      while (seg.next(t, kb0, kb1)) {
        int mb, nb;
        tile_coords(t, num_m, num_n, group, mb, nb);
        for (int kb = kb0; kb < kb1; ++kb) {
          uint8_t* sa = smem + stage * Cfg::STAGE_BYTES;
          const uint32_t lead_full = mapa_shared(smem_u32(&full[stage]), 0);
          if (n_issued >= n_pre) {  // (the first n_pre slots are free and already expect their bytes)
            if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err, CORA_DERR_TMA_WAIT)) goto producer_done;
            if (leader) mbar_arrive_expect_tx(&full[stage], 2 * Cfg::STAGE_BYTES);
            tma_load_2d_pair(sa + Cfg::A_BYTES, &tmB, lead_full, kb * kBK, nb * BN + b_row);
          }
          tma_load_2d_pair(sa, &tmA, lead_full, kb * kBK, mb * 256 + static_cast<int>(rank) * 128);
          ++n_issued;
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    producer_done:;
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      SegIter seg(pair, wsplit);
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
            umma2_bf16(d_tmem, sw128_kmajor_desc(a_addr + k * 32), sw128_kmajor_desc(b_addr + k * 32), IDESC,
                       (kb > kb0 || k > 0) ? 1u : 0u);
          }
          umma2_commit_both(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma2_commit_both(&tfull[acc]);
      }
    }
  } else {
    const int sub = warp & 3;
    const int etid = threadIdx.x - 64;
    const int row_local = sub * 32 + lane;
    const int me = 2 * pair + static_cast<int>(rank);  // this CTA's partial slot / flag
    Stager sg;
    sg.buf[0] = stg + sub * 8192;
    sg.buf[1] = stg + sub * 8192 + 4096;
    sg.cur = 1;
    sg.lane = lane;
    const uint32_t lead_tempty[2] = {mapa_shared(smem_u32(&tempty[0]), 0), mapa_shared(smem_u32(&tempty[1]), 0)};
    int it = 0;
    SegIter seg(pair, wsplit);
    int t, kb0, kb1;
    while (seg.next(t, kb0, kb1)) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      ++it;
      const bool ok = mbar_wait(&tfull[acc], acc_phase, abort_flag, err, CORA_DERR_EPI_WAIT);
      if (named_bar_or(1, 128, !ok)) break;
      tc_fence_after();
      int mb, nb;
      tile_coords(t, num_m, num_n, group, mb, nb);
      const uint32_t tacc = tmem_base + (static_cast<uint32_t>(sub * 32) << 16) + acc * BN;
      const int row0 = mb * 256 + static_cast<int>(rank) * 128 + sub * 32;
      if (ep.split_pair) {
        // Two k-pieces per pair-tile (pair 2t + s): piece s finalises columns
        // [s BN/2, (s+1) BN/2); CTA r of a pair exchanges with CTA r of the other.
        const int s = pair & 1;
        const int other = 2 * (pair ^ 1) + static_cast<int>(rank);
        if (!pair_exchange<BN>(tacc, (1 - s) * (BN / 2), ws.partial + static_cast<int64_t>(me) * kBM * BN,
                               ws.flags + me, ws.flags + other, row_local, etid, abort_flag, err))
          break;
        Partials pp;
        pp.n = 1;
        pp.row = row_local;
        pp.in_smem = false;
        pp.slots[0] = ws.partial + static_cast<int64_t>(other) * kBM * BN;
        gemm_epilogue_warp<BN>(ep, &tmC, tacc, row0, nb * BN, pp, sg, s * (BN / 2), (s + 1) * (BN / 2));
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(lead_tempty[acc]);
        named_bar_sync(1, 128);  // every thread has read the other piece's slot
        if (etid == 0) atomicExch(ws.flags + other, 0);
        continue;
      }
      if (kb0 > 0) {
        // Contributor: hand this CTA's 128-row partial to the tile's finisher.
        float* slot = ws.partial + static_cast<int64_t>(me) * kBM * BN;
        Partials none;
        none.n = 0;
        none.row = row_local;
        none.in_smem = false;
#pragma unroll 1
        for (int c = 0; c < BN; c += 64) {
          float v[4][16];
          const int cols[4] = {c, c + 16, c + 32, c + 48};
          load_acc64(tacc, cols, none, v);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float4* dst = reinterpret_cast<float4*>(slot);
#pragma unroll
            for (int i = 0; i < 4; ++i)
              dst[part_f4(c + 16 * q, i, row_local)] =
                  make_float4(v[q][4 * i], v[q][4 * i + 1], v[q][4 * i + 2], v[q][4 * i + 3]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(lead_tempty[acc]);
        __threadfence();
        named_bar_sync(1, 128);
        if (etid == 0) atomicExch(ws.flags + me, 1);
        continue;
      }
      Partials pp;
      pp.n = 0;
      pp.row = row_local;
      pp.in_smem = false;
      int c_first = 0, c_last = -1;
      if (kb1 < KB) {
        const int last_it = t * KB + KB - 1;
        c_first = pair + 1;
        c_last = c_first;
        while (c_last + 1 < wsplit.G && wsplit.start(c_last + 1) <= last_it) ++c_last;
        const int n_c = c_last - c_first + 1;
        const bool bulk = seg.finished() && n_c * kBM * BN * 4 <= STAGES * Cfg::STAGE_BYTES;
        bool fok = true;
        if (etid == 0) {
          for (int c = c_first; c <= c_last && fok; ++c)
            fok = wait_flag(ws.flags + 2 * c + static_cast<int>(rank), abort_flag, err);
          if (fok && bulk) {
            asm volatile("fence.proxy.async.global;" ::: "memory");
            const uint32_t bytes = kBM * BN * 4;
            mbar_arrive_expect_tx(pbar, bytes * n_c);
            for (int c = c_first; c <= c_last; ++c)
              bulk_g2s(smem + (c - c_first) * bytes,
                       ws.partial + static_cast<int64_t>(2 * c + static_cast<int>(rank)) * kBM * BN, bytes, pbar);
          }
        }
        if (named_bar_or(1, 128, !fok)) break;
        if (bulk) {
          const bool bok = mbar_wait(pbar, pbar_phase, abort_flag, err, CORA_DERR_SPLIT_WAIT);
          pbar_phase ^= 1u;
          if (named_bar_or(1, 128, !bok)) break;
          pp.in_smem = true;
          for (int c = c_first; c <= c_last && pp.n < 4; ++c)
            pp.slots[pp.n++] = reinterpret_cast<const float*>(smem) + static_cast<int64_t>(c - c_first) * kBM * BN;
        } else {
          for (int c = c_first; c <= c_last; ++c) {
            const int slot_id = 2 * c + static_cast<int>(rank);
            (void)ld_acquire(ws.flags + slot_id);
            if (pp.n < 4) pp.slots[pp.n++] = ws.partial + static_cast<int64_t>(slot_id) * kBM * BN;
          }
        }
        if (n_c > 4) record_error(err, CORA_DERR_SPLIT_WAIT);
      }
      gemm_epilogue_warp<BN>(ep, &tmC, tacc, row0, nb * BN, pp, sg);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(lead_tempty[acc]);
      if (c_last >= c_first) {
        named_bar_sync(1, 128);
        if (etid == 0)
          for (int c = c_first; c <= c_last; ++c) atomicExch(ws.flags + 2 * c + static_cast<int>(rank), 0);
      }
    }
    if (lane == 0) bulk_wait_read<0>();  // staging read out (see the 1-CTA kernel)
    __syncwarp();
  }

  // Each warp arrives converged: the producer and MMA warps ran their loops
  // on one lane, and bar.sync counts a divergent warp's lanes separately.
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // no cross-CTA signal is still in flight
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(Cfg::TMEM_COLS)
                 : "memory");
  }
}

}  // namespace cora

namespace cora {

// Failure-detection self-check: one thread waits, with the same bounded waits
// as the GEMM's pipeline, on an mbarrier that nothing arrives at (which = 0)
// or on a flag that nothing sets (which = 1); the wait gives up after
// CORA_WAIT_LIMIT cycles, records its code in `err` and the kernel returns.
__global__ void wait_check_kernel(int which, const int* flag, int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    volatile int* ab = &abort_flag;
    if (which == 0)
      (void)mbar_wait(&bar, 0, ab, err, CORA_DERR_MMA_WAIT);  // phase 0 never completes
    else
      (void)wait_flag(flag, ab, err);  // *flag stays 0
  }
  __syncthreads();
}

}  // namespace cora

using namespace cora;

// The 2-CTA kernel is used for M > 128 unless switched off (cora_gemm_pairs).
static bool g_gemm_pairs_enabled = true;
void gemm_set_pairs(bool on) { g_gemm_pairs_enabled = on; }

int gemm_block_n(int N, int mode) {
  if (mode == CORA_EPI_SWIGLU) return 256;
  return (N % 256 == 0) ? 256 : 128;
}

// Row-tiled kernels: one 128 x 256 fp32 slot per CTA; the few-row kernel:
// two slots of up to 256 x 128 fp32 per CTA.
size_t gemm_workspace_bytes(int num_sms) { return 2 * static_cast<size_t>(num_sms) * kBM * 256 * sizeof(float); }

// A contributor's partial hand-off (epilogue stores, fence, flag) takes about
// as long as 13 k-block MMA steps; skewed equal splits hide it behind the
// finisher's extra k-blocks (skew * S >= 13).
constexpr int kSkewTotal = 14;

// Longest K (in k-blocks) for which the 1-CTA kernel prefers two k-pieces
// sharing the fix-up to three or four skewed pieces (see launch_gemm_bn).
constexpr int kPairMaxKb1 = 128;

// Grid for a stream-K launch: one CTA per SM, but every CTA gets at least
// ceil(KB/4) iterations, so a split tile has at most four contributors
// besides its finisher; never more CTAs than iterations.  Sets the split
// fields of `ep` (uniform unless equal splits apply).
static int gemm_grid(int M, int N, int K, int bn, int num_sms, GemmEpilogue& ep) {
  const int tiles = ((M + kBM - 1) / kBM) * (N / bn);
  const int KB = K / kBK;
  const long long W = static_cast<long long>(tiles) * KB;
  ep.splits = 0;
  ep.split_skew = 0;
  ep.split_pair = 0;
  ep.dp_waves = 0;
  ep.raster_group = 1;
  ep.sk_units = 0;  // set below to the grid
  if (2 * tiles <= num_sms) {
    // Few tiles: split every tile into the same number of k-ranges (at most
    // 4), so each CTA holds one piece and every finisher has its operand
    // ring free for the partial hand-off; skewed toward the finisher.
    int splits = num_sms / tiles;
    if (splits > 4) splits = 4;
    if (splits > KB) splits = KB;
    if (splits == 2 && (ep.mode == CORA_EPI_STORE_BF16 || ep.mode == CORA_EPI_RESID_F32)) {
      // Both pieces share the fix-up, each finalising half of the columns.
      ep.splits = 2;
      ep.split_pair = 1;
    } else if (splits >= 2 && KB % splits == 0) {
      int skew = (kSkewTotal + splits - 1) / splits;
      if (skew > KB / (2 * splits)) skew = KB / (2 * splits);
      ep.splits = splits;
      ep.split_skew = skew;
    }
    ep.sk_units = tiles * splits;
    return tiles * splits;
  }
  long long g = num_sms;
  const long long max_by_share = W / ((KB + 3) / 4);
  if (g > max_by_share) g = max_by_share;
  if (g > W) g = W;
  ep.sk_units = g < 1 ? 1 : static_cast<int>(g);
  return ep.sk_units;
}

// Grid of the 1-CTA kernel: gemm_grid, then two pieces sharing the fix-up
// instead of three or four skewed ones (whose finisher adds three partials),
// unless K is so long that half of it outweighs that: measured at 80-128 rows,
// O (K = 4096) 23.8-24.7 -> 16.6-17.6 us, down (K = 12288) 43.1-43.7 ->
// 45.4-45.9 us.
static int gemm1_grid(int M, int N, int K, int bn, int num_sms, GemmEpilogue& e) {
  int grid = gemm_grid(M, N, K, bn, num_sms, e);
  if (e.splits > 2 && K / kBK <= kPairMaxKb1 && (e.mode == CORA_EPI_STORE_BF16 || e.mode == CORA_EPI_RESID_F32)) {
    const int tiles = grid / e.splits;
    e.splits = 2;
    e.split_skew = 0;
    e.split_pair = 1;
    e.sk_units = tiles * 2;
    grid = tiles * 2;
  }
  return grid;
}

template <int BN>
static cudaError_t launch_gemm_bn(const CUtensorMap& tmA, const CUtensorMap& tmB, const CUtensorMap& tmC, int M,
                                  int N, int K, const GemmEpilogue& ep, const GemmWorkspace& ws, int* err,
                                  int num_sms, cudaStream_t st) {
  using Cfg = GemmCfg<BN>;
  GemmEpilogue e = ep;
  const int grid = gemm1_grid(M, N, K, BN, num_sms, e);
  return launch_pdl(gemm_tc_kernel<BN>, dim3(grid), dim3(192), Cfg::SMEM_BYTES, st, tmA, tmB, tmC, M, N, K, e, ws,
                    err);
}

// Row blocks per group of the tile numbering when a GEMM runs data-parallel
// waves: a wave of 76 pair-tiles then covers 8 row blocks and ~10 weight
// tiles.
constexpr int kRasterGroup = 8;

// Pairs for the 2-CTA kernel: the 1-CTA rule applied to 256 x 256 pair-tiles
// and half the SMs.  With more than two row blocks and at least one tile per
// pair (two row blocks: at least two tiles per pair, e.g. the 512-row gate/up
// projection, 67.6 against 68.0 us and a 0.6 % shorter 256 + 256 decode),
// the tiles run as data-parallel waves over the grouped numbering
// (every pair starts each wave's tile at k-block 0, so the pairs sharing a row
// block or a weight tile read each k-slice of it at about the same time and
// L2 serves all but the first), and only the remainder (tiles mod pairs) is
// split stream-K, first, over as many pairs as give each at least a quarter
// of a tile; the split tiles' hand-offs and fix-ups then run while the pair's
// whole tiles are on the tensor cores.  With one row block, or two and fewer
// than two tiles per pair (the 512-row QKV projection), the M-slowest
// stream-K order already runs the pairs that share a weight tile side by side
// (pair p and p + G/2), and there are too few whole tiles per pair to hide a
// fix-up of up to four partials behind (measured slower).
static int gemm2_pairs(int M, int N, int K, int num_sms, GemmEpilogue& ep) {
  int pairs = gemm_grid(M > 128 ? (M + 1) / 2 : M, N, K, 256, num_sms / 2, ep);
  if (ep.splits > 2 && (ep.mode == CORA_EPI_STORE_BF16 || ep.mode == CORA_EPI_RESID_F32)) {
    // Few pair-tiles (one row block): two pieces sharing the fix-up rather
    // than three or four skewed ones, whose finisher adds three partials.
    const int tiles = pairs / ep.splits;
    ep.splits = 2;
    ep.split_skew = 0;
    ep.split_pair = 1;
    ep.sk_units = tiles * 2;
    pairs = tiles * 2;
  }
  const int num_m = (M + 255) / 256;
  const int tiles = num_m * (N / 256);
  if (ep.splits == 0 && num_m == 1 && tiles <= pairs) {
    // One row block with at most one tile per pair: whole tiles on `tiles`
    // pairs, no partials (QKV at 160-256 rows: 37.2-37.7 -> 26.2-27.7 us
    // against stream-K over every pair with its fix-ups).
    ep.sk_units = tiles;
    return tiles;
  }
  if (ep.splits == 0 && (num_m > 2 || (num_m == 2 && tiles >= 2 * pairs)) && tiles >= pairs) {
    const int KB = K / kBK;
    const int rem = tiles % pairs;
    ep.dp_waves = tiles / pairs;
    ep.raster_group = kRasterGroup;
    ep.sk_units = rem == 0 ? pairs : std::min(pairs, std::max(1, rem * KB / ((KB + 3) / 4)));
  }
  return pairs;
}

cudaError_t launch_wait_check(int which, const int* flag, int* err, cudaStream_t st) {
  wait_check_kernel<<<1, 32, 0, st>>>(which, flag, err);
  return cudaGetLastError();
}

cudaError_t gemm_prepare() {
  cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       GemmCfg<256>::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(gemm_tc2_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, Gemm2Cfg::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(gemm_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              GemmCfg<128>::SMEM_BYTES);
}

cudaError_t launch_gemm(const CUtensorMap& tmA, const CUtensorMap& tmB, const CUtensorMap& tmC, int M, int N, int K,
                        const GemmEpilogue& ep, const GemmWorkspace& ws, int* err, int num_sms, cudaStream_t st) {
  if (gemm_skinny_supported(M, N, K, ep)) {
    CUtensorMap tx;
    if (!make_tmap_bf16_2d(&tx, ep.a_ptr, static_cast<uint64_t>(ep.a_rows), K, static_cast<uint64_t>(K) * 2,
                           gemm_skinny_npad(M), 64))
      return cudaErrorInvalidValue;
    return launch_gemm_skinny(tmB, tx, M, N, K, ep, ws, err, num_sms, st);
  }
  if (M > 128 && N % 256 == 0 && g_gemm_pairs_enabled) {
    GemmEpilogue e = ep;
    const int pairs = gemm2_pairs(M, N, K, num_sms, e);
    return launch_pdl(gemm_tc2_kernel, dim3(2 * pairs), dim3(192), Gemm2Cfg::SMEM_BYTES, st, tmA, tmB, tmC, M, N, K,
                      e, ws, err);
  }
  if (gemm_block_n(N, ep.mode) == 256)
    return launch_gemm_bn<256>(tmA, tmB, tmC, M, N, K, ep, ws, err, num_sms, st);
  return launch_gemm_bn<128>(tmA, tmB, tmC, M, N, K, ep, ws, err, num_sms, st);
}

// Host-side view of how launch_gemm divides an M x N x K projection: the
// kernel it picks and, for the row-tiled kernels, every unit's (CTA or CTA
// pair's) segments in visiting order, as the kernels' own SegIter walks them
// (no device work).  seg: [cap][6] = unit, tile, kb0, kb1, row block, column
// block.  Returns the number of segments (all of them, even beyond cap).
int gemm_plan(int M, int N, int K, int mode, int num_sms, int* info, int* seg, int cap) {
  GemmEpilogue ep{};
  ep.mode = mode;
  ep.head_dim = 128;  // (the few-row kernel's RoPE check; every workload here has head_dim 64 or 128)
  static const uint16_t probe = 0;
  ep.a_ptr = &probe;  // only its presence matters to the few-row kernel's check
  int kind, units, num_m, num_n, group = 1, dp = 0;
  if (gemm_skinny_supported(M, N, K, ep)) {
    info[0] = 0;
    for (int i = 1; i < 7; ++i) info[i] = 0;
    return 0;
  }
  const int KB = K / kBK;
  int W;
  if (M > 128 && N % 256 == 0 && g_gemm_pairs_enabled) {
    kind = 2;
    units = gemm2_pairs(M, N, K, num_sms, ep);
    num_m = (M + 255) / 256;
    num_n = N / 256;
    group = ep.raster_group;
    dp = ep.dp_waves;
    W = (num_m * num_n - dp * units) * KB;
  } else {
    kind = 1;
    const int bn = gemm_block_n(N, mode);
    units = gemm1_grid(M, N, K, bn, num_sms, ep);
    num_m = (M + kBM - 1) / kBM;
    num_n = N / bn;
    W = num_m * num_n * KB;
    ep.sk_units = units;
  }
  info[0] = kind;
  info[1] = units;
  info[2] = num_m * num_n;
  info[3] = KB;
  info[4] = ep.splits;
  info[5] = ep.split_pair;
  info[6] = dp;
  const WorkSplit ws{ep.sk_units, W, KB, ep.splits, ep.split_skew, dp, units};
  int n = 0;
  for (int u = 0; u < units; ++u) {
    SegIter it(u, ws);
    int t, kb0, kb1;
    while (it.next(t, kb0, kb1)) {
      if (n < cap) {
        int mb, nb;
        tile_coords(t, num_m, num_n, group, mb, nb);
        int* r = seg + 6 * n;
        r[0] = u;
        r[1] = t;
        r[2] = kb0;
        r[3] = kb1;
        r[4] = mb;
        r[5] = nb;
      }
      ++n;
    }
  }
  return n;
}

__global__ void rope_transpose_kernel(const float2* __restrict__ rope, float2* __restrict__ rope_t, int seq, int half) {
  const int64_t n = static_cast<int64_t>(seq) * half;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t j = i / seq, p = i - j * seq;  // output index i = j * seq + p
    rope_t[i] = rope[p * half + j];
  }
}

void launch_rope_transpose(const float* rope, float* rope_t, int seq, int half, cudaStream_t st) {
  const int64_t n = static_cast<int64_t>(seq) * half;
  const int blocks = static_cast<int>(std::min<int64_t>((n + 255) / 256, 1024));
  rope_transpose_kernel<<<blocks, 256, 0, st>>>(reinterpret_cast<const float2*>(rope), reinterpret_cast<float2*>(rope_t),
                                                seq, half);
}

// Output tensor map of a GEMM: 32-row x 128-byte boxes, 128-byte swizzle
// (bf16 [M, ldc] for STORE/ROPE/SWIGLU, fp32 [M, ldc] for RESID).
bool make_gemm_out_tmap(CUtensorMap* map, void* C, int M, int ldc, int mode) {
  const bool f32 = mode == CORA_EPI_RESID_F32;
  return make_tmap_2d(map, C, f32 ? 4 : 2, M, ldc, static_cast<uint64_t>(ldc) * (f32 ? 4 : 2), 32, f32 ? 32 : 64);
}
