// Eq. 1 reduction from materialised logits, and the transfer rule + residual
// gate (Eq. 2-4) with block termination, one warp per block of positions.
#include <float.h>
#include <limits.h>

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
// Block (c, row) reduces logits[row, c*chunk : (c+1)*chunk] into one partial.
__global__ void __launch_bounds__(256) reduce_top1_parts_kernel(const uint16_t* __restrict__ logits, int rows, int V,
                                                                int chunk, Top1Part* __restrict__ parts) {
  const int row = blockIdx.y, c = blockIdx.x;
  const int lo = c * chunk;
  const int hi = min(V, lo + chunk);
  const uint16_t* p = logits + static_cast<int64_t>(row) * V;
  Top1 st = top1_empty();
  if ((V & 7) == 0) {
    for (int i = lo + threadIdx.x * 8; i < hi; i += blockDim.x * 8) {
      const uint4 u = __ldcs(reinterpret_cast<const uint4*>(p + i));
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
      float v[8];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        v[2 * j] = __uint_as_float(w[j] << 16);
        v[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
      }
      float mv = v[0];
      int mi = 0;
#pragma unroll
      for (int j = 1; j < 8; ++j)
        if (v[j] > mv) {
          mv = v[j];
          mi = j;
        }
      if (mv > st.m) {
        st.s *= exp2f((st.m - mv) * kLog2e);
        st.m = mv;
        st.idx = i + mi;
      }
      float acc = 0.f;
#pragma unroll
      for (int j = 0; j < 8; ++j) acc += exp2f((v[j] - st.m) * kLog2e);
      st.s += acc;
    }
  } else {
    for (int i = lo + threadIdx.x; i < hi; i += blockDim.x) {
      const float v = bf16_bits_to_float(p[i]);
      if (v > st.m) {
        st.s *= exp2f((st.m - v) * kLog2e);
        st.m = v;
        st.idx = i;
      }
      st.s += exp2f((v - st.m) * kLog2e);
    }
  }
  st = warp_merge(st);
  __shared__ Top1 wpart[8];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) wpart[warp] = st;
  __syncthreads();
  if (warp == 0) {
    st = lane < static_cast<int>(blockDim.x >> 5) ? wpart[lane] : top1_empty();
    st = warp_merge(st);
    if (lane == 0) parts[static_cast<int64_t>(c) * rows + row] = Top1Part{st.m, st.s, st.idx};
  }
}

__device__ __forceinline__ Top1 combine_parts(const Top1Part* __restrict__ parts, int n_parts, int rows, int row) {
  Top1 st = top1_empty();
  for (int q = 0; q < n_parts; ++q) {
    const Top1Part pp = parts[static_cast<int64_t>(q) * rows + row];
    st = top1_merge(st, Top1{pp.m, pp.s, pp.idx});
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
    const Top1Part pp = parts[static_cast<int64_t>(q) * rows + row];
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

// Standalone gate on [B, R] buffers; conf/argmax come from `parts` when given,
// else from conf_in / argmax_in.
__global__ void gate_transfer_kernel(const Top1Part* __restrict__ parts, int n_parts,
                                     const float* __restrict__ conf_in, const int32_t* __restrict__ argmax_in,
                                     float* __restrict__ conf_out, int32_t* __restrict__ argmax_out, int32_t* prev,
                                     int32_t* persist, uint8_t* state, int32_t* tokens, int B, int R, int k,
                                     float tau, int K, uint8_t* unmask, uint8_t* accept, uint8_t* done) {
  const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (b >= B) return;  // warp-uniform
  const int lane = threadIdx.x & 31;
  const bool valid = lane < R;
  const int64_t e = static_cast<int64_t>(b) * R + lane;
  GateLane g{};
  if (valid) {
    if (parts) {
      const Top1 st = combine_parts(parts, n_parts, B * R, static_cast<int>(e));
      g.c = 1.f / st.s;
      g.xhat = st.idx;
      if (conf_out) conf_out[e] = g.c;
      if (argmax_out) argmax_out[e] = g.xhat;
    } else {
      g.c = conf_in[e];
      g.xhat = argmax_in[e];
    }
    g.prev = prev[e];
    g.persist = persist[e];
    g.state = state[e];
    g.token = tokens[e];
  }
  const bool blk_done = gate_warp(g, valid, k, tau, K);
  if (valid) {
    prev[e] = g.prev;
    persist[e] = g.persist;
    state[e] = static_cast<uint8_t>(g.state);
    tokens[e] = g.token;
    unmask[e] = g.T;
    accept[e] = g.A;
  }
  if (lane == 0) done[b] = blk_done;
}

// Session gate: one CTA, warps stride over sequences.  Each unfinished
// sequence combines its LM-head partials (Eq. 1), runs the gate on its active
// block, counts the pass, and on block termination moves to the next block
// with fresh persistence state.  Thread 0 then publishes all_done.
__global__ void session_gate_kernel(SessionGateArgs a) {
  const int lane = threadIdx.x & 31;
  const int nw = blockDim.x >> 5;
  const int n_blocks = a.G / a.BL;
  const int R = a.B * a.BL;
  // Eq. 1: every warp combines whole rows' partials (rows of finished
  // sequences included; they are ignored below).
  for (int r = threadIdx.x >> 5; r < R; r += nw) {
    const Top1 st = warp_combine_parts(a.parts, a.n_parts, R, r);
    if (lane == 0) {
      a.conf[r] = 1.f / st.s;
      a.argmax[r] = st.idx;
    }
  }
  __syncthreads();
  for (int b = threadIdx.x >> 5; b < a.B; b += nw) {
    int32_t* ctrl = a.ctrl + b * 4;
    if (ctrl[3]) continue;  // finished: nothing to do (warp-uniform)
    const int blk = ctrl[0], step = ctrl[1];
    const bool valid = lane < a.BL;
    const int r = b * a.BL + lane;
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
    const int base = a.BL / a.T, extra = a.BL % a.T;
    const int k = base + (step < extra ? 1 : 0);  // transfer schedule
    const bool blk_done = gate_warp(g, valid, k, a.tau, a.K);
    if (valid) {
      a.state[gpos] = static_cast<uint8_t>(g.state);
      a.tokens[cpos] = g.token;
      a.unmask[r] = g.T;
      a.accept[r] = g.A;
      a.prev[r] = blk_done ? -1 : g.prev;      // fresh state for the next block
      a.persist[r] = blk_done ? 0 : g.persist;
    }
    __syncwarp();
    if (lane == 0) {
      ctrl[2] += 1;  // executed passes of this sequence
      if (blk_done) {
        ctrl[0] = blk + 1;
        ctrl[1] = 0;
        if (blk + 1 >= n_blocks) ctrl[3] = 1;
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
  if (threadIdx.x == 0) {
    uint8_t all = 1;
    for (int b = 0; b < a.B; ++b) all &= static_cast<uint8_t>(a.ctrl[b * 4 + 3] != 0);
    *a.all_done = all;
  }
}

}  // namespace cora

using namespace cora;

int reduce_top1_parts_count(int rows, int V, int num_sms) {
  int want = (4 * num_sms + rows - 1) / rows;    // about four CTAs per SM in total
  int max_chunks = (V + 4095) / 4096;            // at least 4096 elements per CTA
  int n = want < max_chunks ? want : max_chunks;
  return n < 1 ? 1 : n;
}

void launch_reduce_top1_parts(const uint16_t* logits, int rows, int V, int n_chunks, Top1Part* parts,
                              cudaStream_t st) {
  int chunk = (V + n_chunks - 1) / n_chunks;
  chunk = (chunk + 7) / 8 * 8;
  dim3 grid(n_chunks, rows);
  reduce_top1_parts_kernel<<<grid, 256, 0, st>>>(logits, rows, V, chunk, parts);
}

void launch_combine_top1(const Top1Part* parts, int n_parts, int rows, float* conf, int32_t* argmax,
                         cudaStream_t st) {
  combine_top1_kernel<<<(rows + 7) / 8, 256, 0, st>>>(parts, n_parts, rows, conf, argmax);
}

void launch_gate_transfer(const Top1Part* parts, int n_parts, const float* conf_in, const int32_t* argmax_in,
                          float* conf_out, int32_t* argmax_out, int32_t* prev, int32_t* persist, uint8_t* state,
                          int32_t* tokens, int B, int R, int k, float tau, int K, uint8_t* unmask, uint8_t* accept,
                          uint8_t* done, cudaStream_t st) {
  const int warps_per_block = 4;
  gate_transfer_kernel<<<(B + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0, st>>>(
      parts, n_parts, conf_in, argmax_in, conf_out, argmax_out, prev, persist, state, tokens, B, R, k, tau, K,
      unmask, accept, done);
}

void launch_session_gate(const SessionGateArgs& a, cudaStream_t st) {
  const int R = a.B * a.BL;
  const int warps = R < 32 ? R : 32;
  session_gate_kernel<<<1, 32 * warps, 0, st>>>(a);
}
