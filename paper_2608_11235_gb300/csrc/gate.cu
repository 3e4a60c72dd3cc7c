// Eq. 1 reduction from materialised logits, and the transfer rule + residual
// gate (Eq. 2-4) with block termination, one warp per block of positions.
#include <float.h>
#include <limits.h>

#include <cudaTypedefs.h>

#include <mutex>

#include "cora_device.cuh"
#include "cora_kernels.h"
#include "../../include/cora.h"

namespace cora {

constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ Top1 top1_empty() { return Top1{-INFINITY, 0.f, INT_MAX}; }

__device__ __forceinline__ Top1 warp_merge(Top1 st) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    Top1 other;
    other.m = __shfl_xor_sync(0xffffffffu, st.m, o);
    other.s = __shfl_xor_sync(0xffffffffu, st.s, o);
    other.idx = __shfl_xor_sync(0xffffffffu, st.idx, o);
    st = top1_merge(st, other);
  }
  return st;
}

// ---------------------------------------------------------------- Eq. 1 (K9)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Adds 8 bf16 logits (one 16-byte word, ids i0 .. i0+7) to a running Top1
// state.  The running max changes rarely, so the common path is a max tree,
// then exp2 terms against the unchanged max.
__device__ __forceinline__ void top1_add8(Top1& st, uint4 u, int i0) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
  float v[8];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    v[2 * j] = __uint_as_float(w[j] << 16);
    v[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
  }
  const float mv = fmaxf(fmaxf(fmaxf(v[0], v[1]), fmaxf(v[2], v[3])), fmaxf(fmaxf(v[4], v[5]), fmaxf(v[6], v[7])));
  if (mv > st.m) {  // new running max: first id attaining it, rescale the sum
    int mi = 7;
#pragma unroll
    for (int j = 6; j >= 0; --j)
      if (v[j] == mv) mi = j;
    st.s *= ex2_approx((st.m - mv) * kLog2e);
    st.m = mv;
    st.idx = i0 + mi;
  }
  const float mL = st.m * kLog2e;
  float acc = 0.f;
#pragma unroll
  for (int j = 0; j < 8; ++j) acc += ex2_approx(fmaf(v[j], kLog2e, -mL));
  st.s += acc;
}

// Partial of logits[row, lo:hi]; block-wide result valid in thread 0.
__device__ __forceinline__ Top1 reduce_range(const uint16_t* __restrict__ p, int lo, int hi, bool vec) {
  Top1 st = top1_empty();
  if (vec) {
    const uint4* pv = reinterpret_cast<const uint4*>(p);
    const int stride = blockDim.x * 8;
    int i = lo + threadIdx.x * 8;
    if (i + 3 * stride < hi) {
      // Four 16-byte loads per batch; the next batch is loaded before the
      // current one is reduced, so eight are in flight while the exponentials run.
      uint4 a = __ldcs(pv + (i >> 3));
      uint4 b = __ldcs(pv + ((i + stride) >> 3));
      uint4 c = __ldcs(pv + ((i + 2 * stride) >> 3));
      uint4 d = __ldcs(pv + ((i + 3 * stride) >> 3));
      int n = i + 4 * stride;
      for (; n + 3 * stride < hi; n += 4 * stride) {
        const uint4 a2 = __ldcs(pv + (n >> 3));
        const uint4 b2 = __ldcs(pv + ((n + stride) >> 3));
        const uint4 c2 = __ldcs(pv + ((n + 2 * stride) >> 3));
        const uint4 d2 = __ldcs(pv + ((n + 3 * stride) >> 3));
        top1_add8(st, a, i);
        top1_add8(st, b, i + stride);
        top1_add8(st, c, i + 2 * stride);
        top1_add8(st, d, i + 3 * stride);
        a = a2;
        b = b2;
        c = c2;
        d = d2;
        i = n;
      }
      top1_add8(st, a, i);
      top1_add8(st, b, i + stride);
      top1_add8(st, c, i + 2 * stride);
      top1_add8(st, d, i + 3 * stride);
      i = n;
    }
    for (; i < hi; i += stride) top1_add8(st, __ldcs(pv + (i >> 3)), i);
  } else {
    for (int i = lo + threadIdx.x; i < hi; i += blockDim.x) {
      const float v = bf16_bits_to_float(p[i]);
      if (v > st.m) {
        st.s *= ex2_approx((st.m - v) * kLog2e);
        st.m = v;
        st.idx = i;
      }
      st.s += ex2_approx((v - st.m) * kLog2e);
    }
  }
  st = warp_merge(st);
  __shared__ Top1 wpart[32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) wpart[warp] = st;
  __syncthreads();
  if (warp == 0) {
    st = lane < static_cast<int>(blockDim.x >> 5) ? wpart[lane] : top1_empty();
    st = warp_merge(st);
  }
  return st;
}

// One warp combines the partials of one row: lane l merges partials l, l+32,
// ... in order, then the lanes merge in a fixed butterfly (deterministic).
__device__ __forceinline__ Top1 warp_combine_parts(const Top1Part* __restrict__ parts, int n_parts, int rows,
                                                   int row) {
  const int lane = threadIdx.x & 31;
  Top1 st = top1_empty();
  for (int q = lane; q < n_parts; q += 32) {
    const Top1Part* src = parts + static_cast<int64_t>(q) * rows + row;
    const Top1Part pp{__ldcg(&src->m), __ldcg(&src->s), __ldcg(&src->idx)};
    st = top1_merge(st, Top1{pp.m, pp.s, pp.idx});
  }
  return warp_merge(st);
}

__global__ void combine_top1_kernel(const Top1Part* __restrict__ parts, int n_parts, int rows,
                                    float* __restrict__ conf, int32_t* __restrict__ argmax) {
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (row >= rows) return;  // warp-uniform
  const Top1 st = warp_combine_parts(parts, n_parts, rows, row);
  if ((threadIdx.x & 31) == 0) {
    conf[row] = 1.f / st.s;  // max_v softmax = exp(m - m) / sum exp(l - m)
    argmax[row] = st.idx;
  }
}

// ------------------------------------------------------------ Eq. 2-4 (K10)
// One warp, lane i = position i of the block (valid when i < R).  Applies
// Eq. 2 to unresolved positions, fixes the min(k, |U|) unresolved positions of
// highest confidence (ties: lower position), accepts the rest when
// c >= tau and m >= K (Eq. 3), and writes tokens/state (Eq. 4).  Returns
// whether the block has no unresolved position left.
struct GateLane {
  float c;
  int xhat;
  int prev;
  int persist;
  int state;
  int token;
  bool T;
  bool A;
};

__device__ __forceinline__ bool gate_warp(GateLane& g, bool valid, int k, float tau, int K) {
  const int lane = threadIdx.x & 31;
  const bool U = valid && g.state == CORA_UNRESOLVED;
  if (U) {
    g.persist = (g.prev == g.xhat) ? g.persist + 1 : 0;  // Eq. 2
    g.prev = g.xhat;
  }
  const unsigned ballot_u = __ballot_sync(0xffffffffu, U);
  const int kk = min(k, __popc(ballot_u));
  int rank = 0;  // unresolved positions ranked ahead of this one
#pragma unroll 4
  for (int j = 0; j < 32; ++j) {
    const float cj = __shfl_sync(0xffffffffu, g.c, j);
    if (((ballot_u >> j) & 1u) && (cj > g.c || (cj == g.c && j < lane))) ++rank;
  }
  g.T = U && rank < kk;                                          // transfer rule
  g.A = U && !g.T && K >= 0 && g.c >= tau && g.persist >= K;     // Eq. 3 on U \ T
  if (g.T) {
    g.token = g.xhat;
    g.state = CORA_TRANSFERRED;
  } else if (g.A) {
    g.token = g.xhat;
    g.state = CORA_ACCEPTED;
  }
  return __ballot_sync(0xffffffffu, valid && g.state == CORA_UNRESOLVED) == 0u;
}

// Gate of block b on [B, R] buffers by one warp (conf/argmax already known).
__device__ __forceinline__ void gate_block(const GateBuffers& gb, int b, int R, int k, float tau, int K) {
  const int lane = threadIdx.x & 31;
  const bool valid = lane < R;
  const int64_t e = static_cast<int64_t>(b) * R + lane;
  GateLane g{};
  if (valid) {
    g.c = gb.conf[e];
    g.xhat = gb.argmax[e];
    g.prev = gb.prev[e];
    g.persist = gb.persist[e];
    g.state = gb.state[e];
    g.token = gb.tokens[e];
  }
  const bool blk_done = gate_warp(g, valid, k, tau, K);
  if (valid) {
    gb.prev[e] = g.prev;
    gb.persist[e] = g.persist;
    gb.state[e] = static_cast<uint8_t>(g.state);
    gb.tokens[e] = g.token;
    gb.unmask[e] = g.T;
    gb.accept[e] = g.A;
  }
  if (lane == 0) gb.done[b] = blk_done;
}

// Standalone gate on [B, R] buffers (conf/argmax given), one warp per block.
__global__ void gate_transfer_kernel(GateBuffers gb, int B, int R, int k, float tau, int K) {
  const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (b >= B) return;  // warp-uniform
  gate_block(gb, b, R, k, tau, K);
}

// Eq. 1 over logits [rows, V] in chunks, fused with what follows.  Block
// (c, row) reduces one chunk to a partial; the last block to finish a group
// (a row, or with the gate a whole block of R rows) combines the group's
// partials in chunk order and then either writes conf/argmax (gate == false)
// or also runs the transfer rule and Eq. 2-4 for that block.  Completion is
// counted with one atomic per block (no waiting); the last block resets the
// counter, so consecutive launches reuse it.
__global__ void __launch_bounds__(256) reduce_fused_kernel(const uint16_t* __restrict__ logits, int rows, int V,
                                                           int chunk, int n_chunks, Top1Part* __restrict__ parts,
                                                           int* __restrict__ counters, GateBuffers gb, int R, int k,
                                                           float tau, int K, int gate) {
  const int row = blockIdx.y, c = blockIdx.x;
  const int lo = c * chunk;
  const int hi = min(V, lo + chunk);
  const Top1 st = reduce_range(logits + static_cast<int64_t>(row) * V, lo, hi, (V & 7) == 0);
  __shared__ int is_last;
  if (threadIdx.x == 0) {
    parts[static_cast<int64_t>(c) * rows + row] = Top1Part{st.m, st.s, st.idx};
    __threadfence();
    const int grp = gate ? row / R : row;
    const int total = gate ? R * n_chunks : n_chunks;
    const int old = atomicAdd(counters + grp, 1);
    is_last = old == total - 1;
    if (is_last) counters[grp] = 0;
  }
  __syncthreads();
  if (!is_last) return;  // uniform per block
  __threadfence();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  if (!gate) {
    if (warp == 0) {
      const Top1 t = warp_combine_parts(parts, n_chunks, rows, row);
      if (lane == 0) {
        gb.conf[row] = 1.f / t.s;  // max_v softmax = exp(m - m) / sum exp(l - m)
        gb.argmax[row] = t.idx;
      }
    }
    return;
  }
  const int b = row / R;
  for (int r = warp; r < R; r += nw) {
    const Top1 t = warp_combine_parts(parts, n_chunks, rows, b * R + r);
    if (lane == 0) {
      gb.conf[b * R + r] = 1.f / t.s;
      gb.argmax[b * R + r] = t.idx;
    }
  }
  __threadfence_block();
  __syncthreads();
  if (warp == 0) gate_block(gb, b, R, k, tau, K);
}

// Session gate: one CTA, warps stride over sequences.  Each unfinished
// sequence combines its LM-head partials (Eq. 1), runs the gate on its active
// block, counts the pass, and on block termination moves to the next block
// with fresh persistence state.  Thread 0 then publishes all_done.
__global__ void session_gate_kernel(SessionGateArgs a) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int nw = blockDim.x >> 5;
  const int n_blocks = a.G / a.BL;
  const int Re = a.B * a.rows_per_seq;
  const bool carry = a.rows_per_seq != a.BL;
  // Eq. 1: every warp combines whole rows' partials (rows of finished
  // sequences included; they are ignored below).
  for (int r = threadIdx.x >> 5; r < Re; r += nw) {
    const int c = r / a.chunk_rows, lr = r - c * a.chunk_rows;
    const int rows_c = min(a.chunk_rows, Re - c * a.chunk_rows);
    const Top1 st =
        warp_combine_parts(a.parts + static_cast<int64_t>(c) * a.n_parts * a.chunk_rows, a.n_parts, rows_c, lr);
    if (lane == 0) {
      a.conf[r] = 1.f / st.s;
      a.argmax[r] = st.idx;
    }
  }
  __syncthreads();
  for (int b = threadIdx.x >> 5; b < a.B; b += nw) {
    int32_t* ctrl = a.ctrl + b * 4;
    if (ctrl[3] || (a.lockstep && ctrl[1] < 0)) {
      // finished, or (prefix cache) block ended and waiting for the other
      // sequences: nothing to do (warp-uniform); no unresolved position left
      if (lane == 0) a.blk_done[b] = 1;
      continue;
    }
    const int blk = ctrl[0], step = ctrl[1];
    if (carry) {
      // Carry-over persistence: Eq. 2 for every unresolved generation
      // position outside the active block (the block's own are updated by
      // the gate below).
      for (int j = lane; j < a.G; j += 32) {
        if (j >= blk * a.BL && j < (blk + 1) * a.BL) continue;
        if (a.state[static_cast<int64_t>(b) * a.G + j] != CORA_UNRESOLVED) continue;
        const int rj = b * a.G + j;
        const int32_t xh = a.argmax[rj];
        a.persist[rj] = a.prev[rj] == xh ? a.persist[rj] + 1 : 0;
        a.prev[rj] = xh;
      }
    }
    const bool valid = lane < a.BL;
    const int r = b * a.rows_per_seq + (carry ? blk * a.BL : 0) + lane;  // Eq. 1 / Eq. 2 row
    const int ru = b * a.BL + lane;                                       // T / A indicator row
    const int64_t cpos = static_cast<int64_t>(b) * a.S + a.P + static_cast<int64_t>(blk) * a.BL + lane;
    const int64_t gpos = static_cast<int64_t>(b) * a.G + static_cast<int64_t>(blk) * a.BL + lane;
    GateLane g{};
    if (valid) {
      g.c = a.conf[r];
      g.xhat = a.argmax[r];
      g.prev = a.prev[r];
      g.persist = a.persist[r];
      g.state = a.state[gpos];
      g.token = a.tokens[cpos];
    }
    int k;
    if (a.schedule == CORA_SCHEDULE_REMAINING) {
      // ceil(|U| / (T - s)) over the block's positions unresolved now
      const int n_u = __popc(__ballot_sync(0xffffffffu, valid && g.state == CORA_UNRESOLVED));
      k = (n_u + (a.T - step) - 1) / (a.T - step);
    } else {
      const int base = a.BL / a.T, extra = a.BL % a.T;
      k = base + (step < extra ? 1 : 0);  // transfer schedule of the block length
    }
    const bool blk_done = gate_warp(g, valid, k, a.tau, a.K);
    if (valid) {
      a.state[gpos] = static_cast<uint8_t>(g.state);
      a.tokens[cpos] = g.token;
      a.unmask[ru] = g.T;
      a.accept[ru] = g.A;
      a.prev[r] = blk_done && !carry ? -1 : g.prev;  // block mode: fresh state for the next block
      a.persist[r] = blk_done && !carry ? 0 : g.persist;
    }
    // EOS-aware stop: a terminated block holding the EOS id ends the sequence;
    // every later generation position takes the EOS id (state EOS_FILLED).
    const bool eos_stop =
        blk_done && a.eos_id >= 0 && __any_sync(0xffffffffu, valid && g.token == a.eos_id) && blk + 1 < n_blocks;
    if (eos_stop) {
      for (int i = (blk + 1) * a.BL + lane; i < a.G; i += 32) {
        a.tokens[static_cast<int64_t>(b) * a.S + a.P + i] = a.eos_id;
        a.state[static_cast<int64_t>(b) * a.G + i] = CORA_EOS_FILLED;
      }
    }
    __syncwarp();
    if (lane == 0) {
      a.blk_done[b] = blk_done ? 1 : 0;
      ctrl[2] += 1;  // executed passes of this sequence
      if (blk_done && a.lockstep && !eos_stop && blk + 1 < n_blocks) {
        ctrl[1] = -1;  // wait: the sequences move to the next block together
      } else if (blk_done) {
        ctrl[0] = blk + 1;
        ctrl[1] = 0;
        if (blk + 1 >= n_blocks || eos_stop) ctrl[3] = 1;
      } else if (step + 1 >= a.T) {
        // The schedule fixes every position by the horizon; reaching it with
        // unresolved positions is an internal error.
        record_error(a.err, CORA_DERR_GATE);
        ctrl[3] = 1;
      } else {
        ctrl[1] = step + 1;
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && a.lockstep) {
    // Once no unfinished sequence is still working on the block, all move on;
    // the next pass is then the new block's first (dense) pass.
    bool active = false, waiting = false;
    int blk = 0;
    for (int b = 0; b < a.B; ++b) {
      const int32_t* c = a.ctrl + b * 4;
      if (c[3]) continue;
      blk = c[0];
      if (c[1] < 0)
        waiting = true;
      else
        active = true;
    }
    int dense_next = 0;
    if (waiting && !active) {
      for (int b = 0; b < a.B; ++b) {
        int32_t* c = a.ctrl + b * 4;
        if (!c[3] && c[1] < 0) {
          c[0] += 1;
          c[1] = 0;
        }
      }
      blk += 1;
      dense_next = 1;
    }
    reinterpret_cast<int32_t*>(a.all_done)[3] = dense_next | (blk << 1);
  }
  if (threadIdx.x == 0) {
    uint8_t all = 1;
    for (int b = 0; b < a.B; ++b) all &= static_cast<uint8_t>(a.ctrl[b * 4 + 3] != 0);
    *a.all_done = all;
  }
}

// Disagreement with the dense endpoint (Sec. 4), one CTA per sequence:
// out[b] = {positions accepted by the gate, of those the ones whose token
// differs from the dense endpoint's, generation positions that differ}.
__global__ void disagreement_kernel(const int32_t* __restrict__ tok, const uint8_t* __restrict__ state,
                                    const int32_t* __restrict__ ref, int S, int P, int G, long long* out) {
  const int b = blockIdx.x;
  int n[3] = {0, 0, 0};
  for (int i = threadIdx.x; i < G; i += blockDim.x) {
    const int64_t c = static_cast<int64_t>(b) * S + P + i;
    const bool diff = tok[c] != ref[c];
    const bool acc = state[static_cast<int64_t>(b) * G + i] == CORA_ACCEPTED;
    n[0] += acc;
    n[1] += acc && diff;
    n[2] += diff;
  }
  __shared__ int red[3][32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
  for (int q = 0; q < 3; ++q) {
    int v = n[q];
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) red[q][w] = v;
  }
  __syncthreads();
  if (threadIdx.x < 3) {
    long long t = 0;
    for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) t += red[threadIdx.x][i];
    out[b * 3 + threadIdx.x] = t;
  }
}

// Loop control of the whole-decode graph (a conditional WHILE node around
// one step): counts the pass in status[2] and keeps looping while some
// sequence is unfinished, no kernel has recorded an error and the horizon
// (n_blocks * T passes) is not reached.
__global__ void step_loop_cond_kernel(cudaGraphConditionalHandle h, int32_t* status, int32_t max_iters) {
  const int32_t it = status[2] + 1;
  status[2] = it;
  const bool done = reinterpret_cast<const uint8_t*>(status)[0] != 0;
  cudaGraphSetConditional(h, (!done && status[1] == 0 && it < max_iters) ? 1u : 0u);
}

}  // namespace cora

using namespace cora;

int reduce_top1_parts_count(int rows, int V, int num_sms) {
  // Resident 256-thread CTAs per SM (register-limited), looked up once.
  static int per_sm = 0;
  if (per_sm == 0) {
    int b = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, reduce_fused_kernel, 256, 0) != cudaSuccess || b < 1) b = 4;
    per_sm = b;
  }
  int want = (4 * num_sms + rows - 1) / rows;    // about four CTAs per SM in total (one wave)
  const int fit = per_sm * num_sms / rows;       // chunks per row that still run in one wave
  if (fit >= 1 && want > fit) want = fit;        // (8 x 32 rows: 3 chunks = 768 CTAs > 760 slots)
  int max_chunks = (V + 4095) / 4096;            // at least 4096 elements per CTA
  int n = want < max_chunks ? want : max_chunks;
  return n < 1 ? 1 : n;
}

void launch_reduce_fused(const uint16_t* logits, int rows, int V, int n_chunks, Top1Part* parts, int* counters,
                         const GateBuffers& gb, int R, int k, float tau, int K, bool gate, cudaStream_t st) {
  int chunk = (V + n_chunks - 1) / n_chunks;
  chunk = (chunk + 7) / 8 * 8;
  dim3 grid(n_chunks, rows);
  reduce_fused_kernel<<<grid, 256, 0, st>>>(logits, rows, V, chunk, n_chunks, parts, counters, gb, R, k, tau, K,
                                            gate ? 1 : 0);
}

void launch_gate_transfer(const GateBuffers& gb, int B, int R, int k, float tau, int K, cudaStream_t st) {
  const int warps_per_block = 4;
  gate_transfer_kernel<<<(B + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0, st>>>(gb, B, R, k, tau,
                                                                                                       K);
}

void launch_combine_top1(const Top1Part* parts, int n_parts, int rows, float* conf, int32_t* argmax,
                         cudaStream_t st) {
  combine_top1_kernel<<<(rows + 7) / 8, 256, 0, st>>>(parts, n_parts, rows, conf, argmax);
}

void launch_session_gate(const SessionGateArgs& a, cudaStream_t st) {
  const int R = a.B * a.BL;
  const int warps = R < 32 ? R : 32;
  launch_pdl(session_gate_kernel, dim3(1), dim3(32 * warps), 0, st, a);
}

// ----------------------------------------------------------------------------
// Allocation-free Eq. 1 reduction.
//
// Some callers cannot allocate device memory at the moment they need this
// reduction: an application whose memory pool already owns the whole device
// (a cudaMalloc would fail or force it to give memory back), or a
// latency-critical loop that must not enter the allocator (cudaMalloc and
// cudaFree synchronise the device).  cora_reduce_top1_noalloc serves them with
// the fixed array below instead of allocated scratch.
//
// When the array occupies device memory: this file is its own CUDA module,
// and with lazy module loading (the default since CUDA 12.2) a module is put
// on a device the first time one of its kernels or symbols is used there.  So
// the array is reserved on a device at the first use of this file's code on
// that device: the first cora_reduce_top1_noalloc call, or earlier any other
// call whose kernels live here (the gate and Eq. 1 reductions).  From then on
// it stays until the process exits (or its context is destroyed), and calls
// reserve nothing more.  A caller whose memory pool will take the whole device
// therefore makes one call before the pool does.
// ----------------------------------------------------------------------------
#define CORA_NOALLOC_MAX_PARTIALS 65536  // (chunk, row) partial states: 768 KiB
#define CORA_NOALLOC_MAX_ROWS 16384      // completion counters: 64 KiB

struct NoAllocScratch {
  Top1Part parts[CORA_NOALLOC_MAX_PARTIALS];
  int counters[CORA_NOALLOC_MAX_ROWS];
};

static __device__ __align__(256) NoAllocScratch g_noalloc_scratch;

namespace {
std::mutex g_noalloc_mu;
// Device address of the array per device, valid for the context it was looked
// up in: a context destroyed by cudaDeviceReset (or a module reloaded in a new
// context) invalidates it, so it is looked up again when the current
// context's unique id differs.
NoAllocScratch* g_noalloc_dev[64];
unsigned long long g_noalloc_ctx[64];
int g_noalloc_sms[64];
PFN_cuCtxGetCurrent_v4000 g_ctx_current = nullptr;
PFN_cuCtxGetId_v12000 g_ctx_id = nullptr;

// Unique id of the calling thread's current context; false if none is
// current yet or it cannot be read.
bool current_context_id(unsigned long long* id) {
  if (!g_ctx_current || !g_ctx_id) {
    cudaDriverEntryPointQueryResult q1, q2;
    void *f1 = nullptr, *f2 = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f1, 4000, cudaEnableDefault, &q1) != cudaSuccess ||
        cudaGetDriverEntryPointByVersion("cuCtxGetId", &f2, 12000, cudaEnableDefault, &q2) != cudaSuccess ||
        q1 != cudaDriverEntryPointSuccess || q2 != cudaDriverEntryPointSuccess || !f1 || !f2)
      return false;
    g_ctx_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(f1);
    g_ctx_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(f2);
  }
  CUcontext ctx = nullptr;
  if (g_ctx_current(&ctx) != CUDA_SUCCESS || !ctx) return false;
  return g_ctx_id(ctx, id) == CUDA_SUCCESS;
}
}  // namespace

extern "C" int cora_reduce_top1_noalloc(const uint16_t* logits, int32_t rows, int32_t V, float* conf, int32_t* argmax,
                                        void* stream) {
  if (!logits || !conf || !argmax) return cora_set_error(CORA_EINVAL, "cora_reduce_top1_noalloc: NULL pointer");
  if (rows < 1 || V < 1) return cora_set_error(CORA_EINVAL, "cora_reduce_top1_noalloc: rows and V must be >= 1");
  if (rows > CORA_NOALLOC_MAX_ROWS)
    return cora_set_error(CORA_EINVAL, "cora_reduce_top1_noalloc: rows exceeds the fixed scratch (max 16384)");
  if ((V & 7) == 0 && (reinterpret_cast<uintptr_t>(logits) & 15u) != 0)
    return cora_set_error(CORA_EINVAL, "cora_reduce_top1_noalloc: logits must be 16-byte aligned");
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
    return cora_set_error(CORA_ECUDA, "cora_reduce_top1_noalloc: no usable current device");
  NoAllocScratch* scratch = nullptr;
  int num_sms = 0;
  {
    // First call on a device (or in a new context on it): look up where the
    // array lives there (the array's name is only a host-side handle) and the
    // SM count.
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    unsigned long long ctx_id = 0;
    const bool have_ctx = current_context_id(&ctx_id);
    if (!have_ctx || !g_noalloc_dev[dev] || g_noalloc_ctx[dev] != ctx_id) {
      g_noalloc_dev[dev] = nullptr;
      void* p = nullptr;
      // (the runtime makes the device's primary context current here if no
      // context is current yet)
      if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p)
        return cora_set_error(CORA_ECUDA, "cora_reduce_top1_noalloc: cudaGetSymbolAddress failed");
      if (!current_context_id(&ctx_id))
        return cora_set_error(CORA_ECUDA, "cora_reduce_top1_noalloc: cannot read the current context");
      if (cudaDeviceGetAttribute(&g_noalloc_sms[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return cora_set_error(CORA_ECUDA, "cora_reduce_top1_noalloc: cannot read the SM count");
      g_noalloc_dev[dev] = static_cast<NoAllocScratch*>(p);
      g_noalloc_ctx[dev] = ctx_id;
    }
    scratch = g_noalloc_dev[dev];
    num_sms = g_noalloc_sms[dev];
  }
  int n_chunks = reduce_top1_parts_count(rows, V, num_sms);
  const int cap = CORA_NOALLOC_MAX_PARTIALS / rows;  // >= 4 since rows <= 16384
  if (n_chunks > cap) n_chunks = cap;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // The counters must start at zero; completed launches leave them at zero,
  // but the array is shared by every call, so clear this call's range first.
  if (cudaMemsetAsync(scratch->counters, 0, sizeof(int) * rows, st) != cudaSuccess)
    return cora_set_error(CORA_ECUDA, "cora_reduce_top1_noalloc: clearing the counters failed");
  GateBuffers gb{conf, argmax, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr};
  launch_reduce_fused(logits, rows, V, n_chunks, scratch->parts, scratch->counters, gb, 1, 0, 0.f, 0, false, st);
  if (cudaGetLastError() != cudaSuccess)
    return cora_set_error(CORA_ECUDA, "cora_reduce_top1_noalloc: kernel launch failed");
  return CORA_OK;
}

cudaError_t launch_step_loop_cond(cudaGraphConditionalHandle h, int32_t* status, int32_t max_iters, cudaStream_t st) {
  step_loop_cond_kernel<<<1, 1, 0, st>>>(h, status, max_iters);
  return cudaGetLastError();
}

void launch_disagreement(const int32_t* tok, const uint8_t* state, const int32_t* ref, int B, int S, int P, int G,
                         long long* out, cudaStream_t st) {
  disagreement_kernel<<<B, 256, 0, st>>>(tok, state, ref, S, P, G, out);
}
