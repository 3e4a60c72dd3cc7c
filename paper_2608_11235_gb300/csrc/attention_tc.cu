// Bidirectional (non-causal) attention on the 5th-generation tensor cores,
// head_dim 128 or 64.  Work item = (sequence, query head, 128-query tile).
// attention_tc_kernel runs one item per CTA and serves head_dim 64 launches
// and head_dim 128 launches whose items fit on the SMs at once; head_dim 128
// launches with more items than SMs go to the two-query-tile persistent
// kernel (attention_tc2.cu).  Keys and values
// stream through shared memory in 128-key tiles (TMA, double-buffered).
//
// Per key tile j:
//   S_j = Q K_j^T        tcgen05.mma M=128 (queries) x N=128 (keys) x K=128 (hd), TMEM
//   softmax              warps 2..5, one query row per thread: the row of S_j is
//                        read from TMEM once; P_j = exp2(S_j - m) (base 2,
//                        scores pre-scaled by log2(e)/sqrt(hd)) goes to shared
//                        memory as bf16 and the row sum l accumulates
//   O += P_j V_j         tcgen05.mma M=128 x N=128 (hd) x K=128 (keys) into one
//                        TMEM accumulator; V is read as an MN-major operand
//                        straight from its [keys][hd] layout
// The reference m of a row is the first tile's max.  Later tiles are
// exponentiated against it without computing their max; only when a tile's
// row sum would pass 2^64 (a score more than ~64 above m, in log2 units) is
// that tile's max taken and m raised to it where it exceeds m by more than 8
// (then O and l are rescaled in place, after the previous PV has completed)
// and the tile redone.  The final O / l is the same for any choice of m (bf16
// and fp32 keep their relative precision at any scale; 2^64 keeps P, l and O
// far from overflow), so the result is unchanged while the softmax warps skip
// the max and never wait for a PV in the common case.
// Two TMEM buffers for S and two P buffers let the softmax of tile j overlap
// the MMAs of tiles j-1 and j+1.  TMEM: S[0] +0, S[1] +128, O +256.
// K and V buffers are released separately (K_j once QK_j is done, V_j once
// PV_j is), so K_{j+2} streams in while tile j is still in the softmax.
// Warps: 0 = TMA producer, 1 = TMEM allocator + MMA issuer, 2..5 = softmax and
// output.  Keys beyond the sequence end are masked; the output is written by
// TMA through a [sequence][row][column] map, which clips rows beyond the end.
#include <math.h>

#include "cora_device.cuh"
#include "cora_kernels.h"

namespace cora {

namespace attn {
constexpr int QT = 128;          // queries per CTA
constexpr int KT = 128;          // keys per tile
constexpr int COL = 128 * 128;   // 16 KB: one 128-row x 64-element swizzle column of a bf16 operand
// Shared memory for head dim hd: Q, K[2], V[2] of hd/64 columns each, P[2] of two columns (128 keys).
template <int HD>
struct Tile {
  static constexpr int OPND = COL * (HD / 64);
  static constexpr int SMEM = 5 * OPND + 4 * COL + 1024 + 256;
};
constexpr float kRescale = 8.0f; // log2 headroom before the reference max is raised
constexpr float kSumLimit = 0x1p64f;  // row sum of a tile beyond which m is raised
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

// Load 128 consecutive fp32 columns of this warp's 32 TMEM lanes (one lane
// per thread) and wait for them, in one statement so that no register is
// read before the load has landed.
__device__ __forceinline__ void tmem_ld128(uint32_t taddr, uint32_t (&r)[128]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x128.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,%64,%65,%66,%67,%68,%69,%70,%71,%72,%73,%74,%75,%76,%77,%78,%79,%80,%81,%82,%83,%84,%85,%86,%87,%88,%89,%90,%91,%92,%93,%94,%95,%96,%97,%98,%99,%100,%101,%102,%103,%104,%105,%106,%107,%108,%109,%110,%111,%112,%113,%114,%115,%116,%117,%118,%119,%120,%121,%122,%123,%124,%125,%126,%127}, [%128];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63]), "=r"(r[64]), "=r"(r[65]), "=r"(r[66]), "=r"(r[67]), "=r"(r[68]), "=r"(r[69]), "=r"(r[70]), "=r"(r[71]), "=r"(r[72]), "=r"(r[73]), "=r"(r[74]), "=r"(r[75]), "=r"(r[76]), "=r"(r[77]), "=r"(r[78]), "=r"(r[79]), "=r"(r[80]), "=r"(r[81]), "=r"(r[82]), "=r"(r[83]), "=r"(r[84]), "=r"(r[85]), "=r"(r[86]), "=r"(r[87]), "=r"(r[88]), "=r"(r[89]), "=r"(r[90]), "=r"(r[91]), "=r"(r[92]), "=r"(r[93]), "=r"(r[94]), "=r"(r[95]), "=r"(r[96]), "=r"(r[97]), "=r"(r[98]), "=r"(r[99]), "=r"(r[100]), "=r"(r[101]), "=r"(r[102]), "=r"(r[103]), "=r"(r[104]), "=r"(r[105]), "=r"(r[106]), "=r"(r[107]), "=r"(r[108]), "=r"(r[109]), "=r"(r[110]), "=r"(r[111]), "=r"(r[112]), "=r"(r[113]), "=r"(r[114]), "=r"(r[115]), "=r"(r[116]), "=r"(r[117]), "=r"(r[118]), "=r"(r[119]), "=r"(r[120]), "=r"(r[121]), "=r"(r[122]), "=r"(r[123]), "=r"(r[124]), "=r"(r[125]), "=r"(r[126]), "=r"(r[127])
      : "r"(taddr)
      : "memory");
}

// Load 32 consecutive fp32 columns of this warp's 32 TMEM lanes (one lane
// per thread) and wait for them, in one statement so that no register is
// read before the load has landed.
__device__ __forceinline__ void tmem_ld32w(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}

// Store 32 consecutive fp32 columns of this warp's 32 TMEM lanes.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};"
               :
               : "r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
               : "memory");
}

__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, const void* src, int c0, int c1, int c2) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1), "r"(c2)
               : "memory");
}

// One CTA per item (grid = query tiles x heads x sequences): used when the
// items fit on the SMs at once.  (On 128 items at S = 512 it measured 12.6 us
// against 13.5 us for a persistent one-tile-per-item variant, ncu, same command.)
template <int HD>
__global__ void __launch_bounds__(192, 1)
    attention_tc_kernel(const __grid_constant__ CUtensorMap tmQKV, const __grid_constant__ CUtensorMap tmOut, int S,
                        int Hq, int Hkv, int q_start, int* err) {
  using namespace attn;
  constexpr int OPND = Tile<HD>::OPND;
  constexpr int NC = HD / 64;  // swizzle columns of a Q / K / V tile
  // idesc: QK M = 128, N = 128 (keys); PV M = 128, N = hd, B (V) MN-major; bf16 x bf16 -> f32.
  constexpr uint32_t IDESC_QK = idesc_bf16_f32(128, 128);
  constexpr uint32_t IDESC_PV = idesc_bf16_f32(128, HD) | (1u << 16);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK[2] = {smem + OPND, smem + 2 * OPND};
  uint8_t* sV[2] = {smem + 3 * OPND, smem + 4 * OPND};
  uint8_t* sP[2] = {smem + 5 * OPND, smem + 5 * OPND + 2 * COL};
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 5 * OPND + 4 * COL);
  uint64_t* qfull = bars + 0;
  uint64_t* kfull = bars + 1;    // [2] K_j landed
  uint64_t* vfull = bars + 3;    // [2] V_j landed
  uint64_t* kempty = bars + 5;   // [2] QK_j done with K_j
  uint64_t* vempty = bars + 7;   // [2] PV_j done with V_j
  uint64_t* sfull = bars + 9;    // [2] S_j in TMEM
  uint64_t* sfree = bars + 11;   // [2] S_j read out by the four softmax warps
  uint64_t* pfull = bars + 13;   // [2] P_j written (and O rescaled, if it was)
  uint64_t* pdone = bars + 15;   // [2] PV_j complete (P buffer free, O up to date)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 17);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int kvh = h / (Hq / Hkv);
  const int q0 = q_start + qt * QT;  // queries q_start .. ; output rows relative to q_start
  const int row_base = b * S;                       // first row of this sequence in [B*S, .]
  const int n_kt = (S + KT - 1) / KT;
  const int qcol = h * HD, kcol = (Hq + kvh) * HD, vcol = (Hq + Hkv + kvh) * HD;

  if (threadIdx.x == 0) {
    mbar_init(qfull, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kfull[i], 1);
      mbar_init(&vfull[i], 1);
      mbar_init(&kempty[i], 1);
      mbar_init(&vempty[i], 1);
      mbar_init(&sfull[i], 1);
      mbar_init(&sfree[i], 4);
      mbar_init(&pfull[i], 4);
      mbar_init(&pdone[i], 1);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmQKV);
    tma_prefetch_desc(&tmOut);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
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
      mbar_arrive_expect_tx(qfull, OPND);
      for (int c = 0; c < NC; ++c) tma_load_2d(sQ + c * COL, &tmQKV, qfull, qcol + c * 64, row_base + q0);
      for (int j = 0; j < n_kt; ++j) {
        const int s = j & 1;
        const uint32_t ph = ((j >> 1) & 1) ^ 1u;
        const int r = row_base + j * KT;
        if (!mbar_wait(&kempty[s], ph, abort_flag, err, CORA_DERR_TMA_WAIT)) break;
        mbar_arrive_expect_tx(&kfull[s], OPND);
        for (int c = 0; c < NC; ++c) tma_load_2d(sK[s] + c * COL, &tmQKV, &kfull[s], kcol + c * 64, r);
        if (!mbar_wait(&vempty[s], ph, abort_flag, err, CORA_DERR_TMA_WAIT)) break;
        mbar_arrive_expect_tx(&vfull[s], OPND);
        for (int c = 0; c < NC; ++c) tma_load_2d(sV[s] + c * COL, &tmQKV, &vfull[s], vcol + c * 64, r);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = mbar_wait(qfull, 0, abort_flag, err, CORA_DERR_MMA_WAIT);
      const uint32_t q_addr = smem_u32(sQ);
      const uint32_t o_tmem = tmem_base + 256;
      // O += P_jj V_jj.
      auto issue_pv = [&](int jj) -> bool {
        const int s = jj & 1;
        if (!mbar_wait(&pfull[s], (jj >> 1) & 1, abort_flag, err, CORA_DERR_MMA_WAIT)) return false;
        if (!mbar_wait(&vfull[s], (jj >> 1) & 1, abort_flag, err, CORA_DERR_MMA_WAIT)) return false;
        tc_fence_after();
        const uint32_t p_addr = smem_u32(sP[s]), v_addr = smem_u32(sV[s]);
#pragma unroll
        for (int k = 0; k < KT / 16; ++k) {
          // A = P: K-major, keys contiguous, 64-key swizzle columns 16 KB apart.
          const uint64_t a = sw128_kmajor_desc(p_addr + (k >> 2) * COL + (k & 3) * 32);
          // B = V: rows are keys (K), 64-element hd blocks 16 KB apart (MN-major).
          const uint64_t bd = sw128_mnmajor_desc(v_addr + k * 16 * 128, COL);
          umma_bf16(o_tmem, a, bd, IDESC_PV, (jj > 0 || k > 0) ? 1u : 0u);
        }
        umma_commit(&pdone[s]);
        umma_commit(&vempty[s]);
        return true;
      };
      for (int j = 0; ok && j < n_kt; ++j) {
        const int s = j & 1;
        const uint32_t ph = (j >> 1) & 1;
        if (!mbar_wait(&kfull[s], ph, abort_flag, err, CORA_DERR_MMA_WAIT)) break;
        if (!mbar_wait(&sfree[s], ph ^ 1u, abort_flag, err, CORA_DERR_MMA_WAIT)) break;
        tc_fence_after();
        const uint32_t k_addr = smem_u32(sK[s]);
        const uint32_t d = tmem_base + s * 128;
#pragma unroll
        for (int k = 0; k < HD / 16; ++k) {
          const uint32_t off = (k >> 2) * COL + (k & 3) * 32;
          umma_bf16(d, sw128_kmajor_desc(q_addr + off), sw128_kmajor_desc(k_addr + off), IDESC_QK, k > 0);
        }
        umma_commit(&sfull[s]);
        umma_commit(&kempty[s]);
        if (j >= 1 && !issue_pv(j - 1)) break;
      }
      if (ok && n_kt >= 1) issue_pv(n_kt - 1);
    }
  } else {
    const int sub = warp & 3;
    const int r = sub * 32 + lane;  // query row within the tile (TMEM lane)
    const uint32_t lane_base = tmem_base + (static_cast<uint32_t>(sub * 32) << 16);
    const uint32_t o_lane = lane_base + 256;
    const float sl2 = 1.4426950408889634f / sqrtf(static_cast<float>(HD));
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < n_kt && ok; ++j) {
      const int s = j & 1;
      const uint32_t ph = (j >> 1) & 1;
      ok = mbar_wait(&sfull[s], ph, abort_flag, err, CORA_DERR_EPI_WAIT);
      if (!ok) break;
      tc_fence_after();
      uint32_t v[128];
      tmem_ld128(lane_base + s * 128, v);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sfree[s]);  // S buffer may take S_{j+2}
      const int kbase = j * KT;
      if (kbase + KT > S) {  // ragged last tile: keys past the end do not count
#pragma unroll
        for (int i = 0; i < KT; ++i)
          if (kbase + i >= S) v[i] = __float_as_uint(-INFINITY);
      }
      // Exact tile max; raise m where it exceeds m + kRescale (rescaling O
      // after the previous PV).  Returns false on a timed-out wait.
      auto raise_to_max = [&]() -> bool {
        float mx8[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) mx8[i] = -INFINITY;
#pragma unroll
        for (int i = 0; i < KT; ++i) mx8[i & 7] = fmaxf(mx8[i & 7], __uint_as_float(v[i]));
        float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                         fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
        mx *= sl2;
        const bool raise = mx > m + kRescale;
        if (__any_sync(0xffffffffu, raise)) {
          const float m_new = raise ? mx : m;
          const float a = ex2f(m - m_new);
          l *= a;
          m = m_new;
          if (j > 0) {
            const int sp = (j - 1) & 1;
            if (!mbar_wait(&pdone[sp], ((j - 1) >> 1) & 1, abort_flag, err, CORA_DERR_EPI_WAIT)) return false;
            tc_fence_after();
#pragma unroll 1
            for (int c = 0; c < HD; c += 32) {
              uint32_t o[32];
              tmem_ld32w(o_lane + c, o);
#pragma unroll
              for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * a);
              tmem_st32(o_lane + c, o);
            }
            tmem_wait_st();
          }
        }
        return true;
      };
      uint8_t* prow = sP[s];
      auto exp_tile = [&]() -> float {
        float rs4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int c = 0; c < KT; c += 8) {
          uint32_t pk[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float x0 = ex2f(fmaf(__uint_as_float(v[c + 2 * i]), sl2, -m));
            const float x1 = ex2f(fmaf(__uint_as_float(v[c + 2 * i + 1]), sl2, -m));
            rs4[i] += x0 + x1;
            pk[i] = pack_bf16x2(x0, x1);
          }
          const int chunk = (c & 63) >> 3;
          *reinterpret_cast<uint4*>(prow + (c >> 6) * COL + r * 128 + ((chunk ^ (r & 7)) << 4)) =
              make_uint4(pk[0], pk[1], pk[2], pk[3]);
        }
        return (rs4[0] + rs4[1]) + (rs4[2] + rs4[3]);
      };
      if (j == 0) {
        ok = raise_to_max();
        if (!ok) break;
      }
      // P buffer s is free once PV_{j-2} has read it.
      if (j >= 2) ok = mbar_wait(&pdone[s], ph ^ 1u, abort_flag, err, CORA_DERR_EPI_WAIT);
      if (!ok) break;
      // Later tiles are exponentiated against m without their own max; only
      // when a row's sum would pass kSumLimit is the max taken and the tile redone.
      float rs = exp_tile();
      if (j > 0 && __any_sync(0xffffffffu, !(rs <= kSumLimit))) {
        ok = raise_to_max();
        if (!ok) break;
        rs = exp_tile();
      }
      l += rs;
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&pfull[s]);
    }
    // Output: wait for the last PV, O / l as bf16 into this warp's 32 rows of
    // a free P buffer (same swizzled layout as the store map's box), then TMA.
    if (ok) {
      const int sl = (n_kt - 1) & 1;
      ok = mbar_wait(&pdone[sl], ((n_kt - 1) >> 1) & 1, abort_flag, err, CORA_DERR_EPI_WAIT);
    }
    if (ok) {
      tc_fence_after();
      const float inv = 1.f / l;
      uint8_t* stg = sP[0];
#pragma unroll 1
      for (int c0 = 0; c0 < HD; c0 += 32) {
        uint32_t o[32];
        tmem_ld32w(o_lane + c0, o);
#pragma unroll
        for (int i = 0; i < 32; i += 8) {
          const int c = c0 + i;
          const int chunk = (c & 63) >> 3;
          *reinterpret_cast<uint4*>(stg + (c >> 6) * COL + r * 128 + ((chunk ^ (r & 7)) << 4)) = make_uint4(
              pack_bf16x2(__uint_as_float(o[i]) * inv, __uint_as_float(o[i + 1]) * inv),
              pack_bf16x2(__uint_as_float(o[i + 2]) * inv, __uint_as_float(o[i + 3]) * inv),
              pack_bf16x2(__uint_as_float(o[i + 4]) * inv, __uint_as_float(o[i + 5]) * inv),
              pack_bf16x2(__uint_as_float(o[i + 6]) * inv, __uint_as_float(o[i + 7]) * inv));
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        for (int c = 0; c < NC; ++c)
          tma_store_3d(&tmOut, stg + c * COL + sub * 32 * 128, qcol + c * 64, qt * QT + sub * 32, b);
        asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
      }
    }
    tc_fence_before();
  }

  // Each warp arrives converged: the producer and MMA warps ran their loops
  // on one lane, and bar.sync counts a divergent warp's lanes separately.
  __syncwarp();
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
  cudaError_t e = cudaFuncSetAttribute(attention_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       attn::Tile<128>::SMEM);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attention_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              attn::Tile<64>::SMEM);
}

cudaError_t launch_attention_tc(const CUtensorMap& tmQKV, uint16_t* out, int B, int S, int Hq, int Hkv, int hd,
                                int q_start, int q_len, int* err, int num_sms, cudaStream_t st) {
  // Output map [B][q_len][Hq*hd] bf16, boxes of 32 rows x 64 columns (one
  // warp's rows, one 128-byte swizzle column).
  CUtensorMap tmOut;
  if (!make_tmap_bf16_3d(&tmOut, out, static_cast<uint64_t>(Hq) * hd, q_len, B, static_cast<uint64_t>(Hq) * hd * 2,
                         static_cast<uint64_t>(q_len) * Hq * hd * 2, 64, 32, 1))
    return cudaErrorInvalidValue;
  const int n_qt = (q_len + attn::QT - 1) / attn::QT;
  const int n_items = n_qt * Hq * B;
  if (hd == 64)  // one CTA per item, in as many waves as it takes
    return launch_pdl(attention_tc_kernel<64>, dim3(n_qt, Hq, B), dim3(192), attn::Tile<64>::SMEM, st, tmQKV, tmOut,
                      S, Hq, Hkv, q_start, err);
  if (n_items <= num_sms)
    return launch_pdl(attention_tc_kernel<128>, dim3(n_qt, Hq, B), dim3(192), attn::Tile<128>::SMEM, st, tmQKV,
                      tmOut, S, Hq, Hkv, q_start, err);
  // More items than SMs: two query tiles per CTA (attention_tc2.cu).
  return launch_attention_tc2(tmQKV, out, B, S, Hq, Hkv, q_start, q_len, err, num_sms, st);
}
