// Bidirectional (non-causal) attention, head_dim 128, two query tiles per CTA.
//
// Work item = (sequence, query head, pair of 128-query tiles); persistent grid
// of min(items, SMs) CTAs, CTA c taking items c, c + grid, ...  Both query
// tiles of an item read the same 128-key K/V tiles, so every K/V tile brought
// into shared memory serves 256 queries, and the two tiles' softmax streams
// run on separate warpgroups.
//
// Per key tile j and query tile g (g = 0, 1):
//   S_g = Q_g K_j^T     tcgen05.mma M=128 x N=128 x K=128 into TMEM (S_g)
//   softmax             warpgroup g, one query row per thread: the S row is read
//                       from TMEM once; P = exp2(S log2(e)/sqrt(hd) - m) is packed
//                       to bf16 and written back into the first 64 columns of
//                       S_g (tcgen05.st); the row sum l accumulates in fp32
//   O_g += P V_j        tcgen05.mma with A = P read from TMEM, B = V_j from
//                       shared memory (MN-major, straight from [keys][hd])
// One thread issues every MMA, in the order QK_0(0) QK_1(0), then per j:
// PV_0(j) QK_0(j+1) PV_1(j) QK_1(j+1).  tcgen05 MMAs of one thread execute in
// issue order, so QK_g(j+1) overwrites S_g only after PV_g(j) has read P_g(j)
// from it, and the commit after QK_g(j+1) (the softmax's "S ready" signal)
// also means PV_g(j) is complete: O_g may then be rescaled in place.  The
// reference m of a row is the item's first key tile's max; later tiles are
// exponentiated against it without computing their max, and only when a
// tile's row sum would pass 2^64 is its max taken, m raised where it exceeds
// m by more than 8 (O and l rescaled) and the tile redone.  O / l is the same
// for any m (see attention_tc.cu).

// TMEM: S_0 +0, S_1 +128, O_0 +256, O_1 +384 (512 columns).
// Shared memory: Q_0, Q_1, K[2], V[2] (32 KB each).  The output O / l goes from
// registers to global memory (one row per thread), rows past the query range
// skipped.  An item whose second tile lies past the range computes it on
// whatever rows TMA brings (zero fill past the tensor) and stores nothing.
// Warps: 0 = TMA producer, 1 = TMEM allocator + MMA issuer, 2-3 idle,
// 4-7 = softmax of query tile 0, 8-11 = softmax of query tile 1 (a warpgroup
// reads the TMEM lanes 32 * (warp % 4) .. + 31, so each group is 4 aligned warps).
#include <math.h>

#include "cora_device.cuh"
#include "cora_kernels.h"

namespace cora {

namespace attn2 {
constexpr int QT = 128;            // queries per tile
constexpr int KT = 128;            // keys per tile
constexpr int HD = 128;            // head dim
constexpr int OPND = QT * HD * 2;  // 32 KB: one 128 x 128 bf16 operand (two 16 KB swizzle columns)
constexpr int SMEM = 6 * OPND + 1024 + 256;  // Q[2], K[2], V[2]
constexpr int THREADS = 384;
constexpr float kRescale = 8.0f;   // log2 headroom before the reference max is raised
constexpr float kSumLimit = 0x1p64f;  // row sum of a tile beyond which m is raised
}  // namespace attn2

// MN-major (N contiguous) 128-byte-swizzled operand: 8-row K groups 1024 B
// apart (stride byte offset), 64-element N blocks `lbo` bytes apart.
__device__ __forceinline__ uint64_t sw128_mn_desc(uint32_t smem_addr, uint32_t lbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((smem_addr & 0x3FFFF) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFF) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

// D[tmem] (+)= A[tmem] * B[smem], bf16 inputs, fp32 accumulate; A is M x K
// with its rows in TMEM lanes and K along columns (two bf16 per column).
__device__ __forceinline__ void umma_bf16_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                                 uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// 32 consecutive fp32 columns of this warp's 32 TMEM lanes, loaded and waited for.
__device__ __forceinline__ void tm_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}

// 128 consecutive fp32 columns of this warp's 32 TMEM lanes, loaded and waited for.
__device__ __forceinline__ void tm_ld128(uint32_t taddr, uint32_t (&r)[128]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x128.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,%64,%65,%66,%67,%68,%69,%70,%71,%72,%73,%74,%75,%76,%77,%78,%79,%80,%81,%82,%83,%84,%85,%86,%87,%88,%89,%90,%91,%92,%93,%94,%95,%96,%97,%98,%99,%100,%101,%102,%103,%104,%105,%106,%107,%108,%109,%110,%111,%112,%113,%114,%115,%116,%117,%118,%119,%120,%121,%122,%123,%124,%125,%126,%127}, [%128];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63]), "=r"(r[64]), "=r"(r[65]), "=r"(r[66]), "=r"(r[67]), "=r"(r[68]), "=r"(r[69]), "=r"(r[70]), "=r"(r[71]), "=r"(r[72]), "=r"(r[73]), "=r"(r[74]), "=r"(r[75]), "=r"(r[76]), "=r"(r[77]), "=r"(r[78]), "=r"(r[79]), "=r"(r[80]), "=r"(r[81]), "=r"(r[82]), "=r"(r[83]), "=r"(r[84]), "=r"(r[85]), "=r"(r[86]), "=r"(r[87]), "=r"(r[88]), "=r"(r[89]), "=r"(r[90]), "=r"(r[91]), "=r"(r[92]), "=r"(r[93]), "=r"(r[94]), "=r"(r[95]), "=r"(r[96]), "=r"(r[97]), "=r"(r[98]), "=r"(r[99]), "=r"(r[100]), "=r"(r[101]), "=r"(r[102]), "=r"(r[103]), "=r"(r[104]), "=r"(r[105]), "=r"(r[106]), "=r"(r[107]), "=r"(r[108]), "=r"(r[109]), "=r"(r[110]), "=r"(r[111]), "=r"(r[112]), "=r"(r[113]), "=r"(r[114]), "=r"(r[115]), "=r"(r[116]), "=r"(r[117]), "=r"(r[118]), "=r"(r[119]), "=r"(r[120]), "=r"(r[121]), "=r"(r[122]), "=r"(r[123]), "=r"(r[124]), "=r"(r[125]), "=r"(r[126]), "=r"(r[127])
      : "r"(taddr)
      : "memory");
}

// Store 32 consecutive 32-bit columns of this warp's 32 TMEM lanes.
__device__ __forceinline__ void tm_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};"
               :
               : "r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
                 "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
                 "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]),
                 "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
               : "memory");
}

__device__ __forceinline__ void tm_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ float ex2_approx_ftz(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__global__ void __launch_bounds__(attn2::THREADS, 1)
    attention_tc2_kernel(const __grid_constant__ CUtensorMap tmQKV, uint16_t* __restrict__ out, int S, int Hq,
                         int Hkv, int q_start, int q_len, int n_pairs, int n_items, int* err) {
  using namespace attn2;
  // idesc: M = 128, N = 128, bf16 x bf16 -> f32; PV reads B (V) MN-major.
  constexpr uint32_t IDESC_QK = idesc_bf16_f32(128, 128);
  constexpr uint32_t IDESC_PV = idesc_bf16_f32(128, 128) | (1u << 16);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;  // Q_0 at +0, Q_1 at +OPND
  uint8_t* sK[2] = {smem + 2 * OPND, smem + 3 * OPND};
  uint8_t* sV[2] = {smem + 4 * OPND, smem + 5 * OPND};
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 6 * OPND);
  uint64_t* qfull = bars + 0;    // Q_0 and Q_1 of the item landed
  uint64_t* qempty = bars + 1;   // every QK of the item done (Q buffers free)
  uint64_t* kfull = bars + 2;    // [2] K tile landed
  uint64_t* vfull = bars + 4;    // [2] V tile landed
  uint64_t* kempty = bars + 6;   // [2] both QKs done with the K tile
  uint64_t* vempty = bars + 8;   // [2] both PVs done with the V tile
  uint64_t* sfull = bars + 10;   // [2] per query tile: S in TMEM (and the tile's previous PV complete)
  uint64_t* pfull = bars + 12;   // [2] per query tile: P written to TMEM (and O rescaled, if it was)
  uint64_t* odone = bars + 14;   // [2] per query tile: the item's last PV complete
  uint64_t* oempty = bars + 16;  // [2] per query tile: O read out by the softmax warpgroup
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 18);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_kt = (S + KT - 1) / KT;
  const int group = Hq / Hkv;
  // Item -> (query tile pair, query head, sequence), pair fastest.
  auto item_coords = [&](int item, int& pr, int& h, int& b) {
    pr = item % n_pairs;
    const int rest = item / n_pairs;
    h = rest % Hq;
    b = rest / Hq;
  };

  if (threadIdx.x == 0) {
    mbar_init(qfull, 1);
    mbar_init(qempty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kfull[i], 1);
      mbar_init(&vfull[i], 1);
      mbar_init(&kempty[i], 1);
      mbar_init(&vempty[i], 1);
      mbar_init(&sfull[i], 1);
      mbar_init(&pfull[i], 4);
      mbar_init(&odone[i], 1);
      mbar_init(&oempty[i], 4);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) tma_prefetch_desc(&tmQKV);
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
      bool ok = true;
      int t = 0;  // key tiles loaded so far by this CTA (ring slot t & 1)
      for (int it = 0, item = blockIdx.x; ok && item < n_items; ++it, item += gridDim.x) {
        int pr, h, b;
        item_coords(item, pr, h, b);
        const int kvh = h / group;
        const int row_base = b * S;                   // first row of this sequence in [B*S, .]
        const int q0 = q_start + pr * 2 * QT;         // first query of the pair
        const int qcol = h * HD, kcol = (Hq + kvh) * HD, vcol = (Hq + Hkv + kvh) * HD;
        if (it > 0 && !mbar_wait(qempty, (it - 1) & 1, abort_flag, err, CORA_DERR_TMA_WAIT)) break;
        mbar_arrive_expect_tx(qfull, 2 * OPND);
        for (int g = 0; g < 2; ++g) {
          tma_load_2d(sQ + g * OPND, &tmQKV, qfull, qcol, row_base + q0 + g * QT);
          tma_load_2d(sQ + g * OPND + OPND / 2, &tmQKV, qfull, qcol + 64, row_base + q0 + g * QT);
        }
        for (int j = 0; j < n_kt; ++j, ++t) {
          const int s = t & 1;
          const uint32_t ph = ((t >> 1) & 1) ^ 1u;
          const int r = row_base + j * KT;
          if (!mbar_wait(&kempty[s], ph, abort_flag, err, CORA_DERR_TMA_WAIT)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&kfull[s], OPND);
          tma_load_2d(sK[s], &tmQKV, &kfull[s], kcol, r);
          tma_load_2d(sK[s] + OPND / 2, &tmQKV, &kfull[s], kcol + 64, r);
          if (!mbar_wait(&vempty[s], ph, abort_flag, err, CORA_DERR_TMA_WAIT)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&vfull[s], OPND);
          tma_load_2d(sV[s], &tmQKV, &vfull[s], vcol, r);
          tma_load_2d(sV[s] + OPND / 2, &tmQKV, &vfull[s], vcol + 64, r);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t q_addr = smem_u32(sQ);
      // S_g = Q_g K^T for the key tile in ring slot s.
      auto issue_qk = [&](int g, int s) {
        const uint32_t k_addr = smem_u32(sK[s]);
        const uint32_t d = tmem_base + g * 128;
#pragma unroll
        for (int k = 0; k < HD / 16; ++k) {
          const uint32_t off = (k >> 2) * (OPND / 2) + (k & 3) * 32;
          umma_bf16(d, sw128_kmajor_desc(q_addr + g * OPND + off), sw128_kmajor_desc(k_addr + off), IDESC_QK, k > 0);
        }
        umma_commit(&sfull[g]);
      };
      // O_g (+)= P_g V for the value tile in ring slot s; P_g is in the first
      // 64 columns of S_g (16 keys = 8 columns per MMA).
      auto issue_pv = [&](int g, int s, bool first) {
        const uint32_t v_addr = smem_u32(sV[s]);
        const uint32_t o = tmem_base + 256 + g * 128;
#pragma unroll
        for (int k = 0; k < KT / 16; ++k) {
          const uint64_t bd = sw128_mn_desc(v_addr + k * 16 * 128, OPND / 2);
          umma_bf16_tmem_a(o, tmem_base + g * 128 + k * 8, bd, IDESC_PV, (!first || k > 0) ? 1u : 0u);
        }
      };
      bool ok = true;
      int t = 0;  // key tiles of this CTA whose QKs were issued
      for (int it = 0, item = blockIdx.x; ok && item < n_items; ++it, item += gridDim.x) {
        if (!mbar_wait(qfull, it & 1, abort_flag, err, CORA_DERR_MMA_WAIT)) break;
        {
          const int s = t & 1;
          if (!mbar_wait(&kfull[s], (t >> 1) & 1, abort_flag, err, CORA_DERR_MMA_WAIT)) break;
          tc_fence_after();
          issue_qk(0, s);
          issue_qk(1, s);
          umma_commit(&kempty[s]);
          if (n_kt == 1) umma_commit(qempty);
        }
        for (int j = 0; j < n_kt; ++j) {
          const int tt = t + j;  // this key tile's index in the CTA's ring
          const int s = tt & 1, s1 = (tt + 1) & 1;
          const bool last = j == n_kt - 1;
          for (int g = 0; g < 2 && ok; ++g) {
            // PV_g(j): P_g written (softmax g), V landed, and, for an item's
            // first PV, the previous item's O_g read out.
            ok = mbar_wait(&pfull[g], tt & 1, abort_flag, err, CORA_DERR_MMA_WAIT) &&
                 (g == 1 || mbar_wait(&vfull[s], (tt >> 1) & 1, abort_flag, err, CORA_DERR_MMA_WAIT)) &&
                 (j > 0 || mbar_wait(&oempty[g], (it & 1) ^ 1u, abort_flag, err, CORA_DERR_MMA_WAIT));
            if (!ok) break;
            tc_fence_after();
            issue_pv(g, s, j == 0);
            if (g == 1) umma_commit(&vempty[s]);
            if (last) umma_commit(&odone[g]);
            if (!last) {
              // QK_g(j+1) right after PV_g(j): it overwrites S_g (and P_g) only
              // after that PV has read them (MMAs of one thread run in order).
              if (g == 0) {
                ok = mbar_wait(&kfull[s1], ((tt + 1) >> 1) & 1, abort_flag, err, CORA_DERR_MMA_WAIT);
                if (!ok) break;
                tc_fence_after();
              }
              issue_qk(g, s1);
              if (g == 1) {
                umma_commit(&kempty[s1]);
                if (j + 1 == n_kt - 1) umma_commit(qempty);
              }
            }
          }
          if (!ok) break;
        }
        t += n_kt;
      }
    }
  } else if (warp >= 4) {
    const int g = (warp - 4) >> 2;  // query tile of this warpgroup
    const int sub = warp & 3;
    const int r = sub * 32 + lane;  // query row within the tile (TMEM lane)
    const uint32_t lane_base = tmem_base + (static_cast<uint32_t>(sub * 32) << 16);
    const uint32_t s_lane = lane_base + g * 128;
    const uint32_t o_lane = lane_base + 256 + g * 128;
    const float sl2 = 1.4426950408889634f / sqrtf(static_cast<float>(HD));
    const int ldo = Hq * HD;
    bool ok = true;
    int t = 0;  // key tiles this warpgroup has taken
    for (int it = 0, item = blockIdx.x; ok && item < n_items; ++it, item += gridDim.x) {
      int pr, h, b;
      item_coords(item, pr, h, b);
      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < n_kt; ++j, ++t) {
        ok = mbar_wait(&sfull[g], t & 1, abort_flag, err, CORA_DERR_EPI_WAIT);
        if (!ok) break;
        tc_fence_after();
        uint32_t v[128];
        tm_ld128(s_lane, v);
        const int kbase = j * KT;
        if (kbase + KT > S) {  // ragged last tile: keys past the end do not count
#pragma unroll
          for (int i = 0; i < KT; ++i)
            if (kbase + i >= S) v[i] = __float_as_uint(-INFINITY);
        }
        // P = exp2(S * sl2 - m) as bf16 pairs over the first 64 columns of S_g;
        // returns the row sum of this tile.
        auto exp_tile = [&]() -> float {
          float rs4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            uint32_t pk[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float x0 = ex2_approx_ftz(fmaf(__uint_as_float(v[64 * half + 2 * i]), sl2, -m));
              const float x1 = ex2_approx_ftz(fmaf(__uint_as_float(v[64 * half + 2 * i + 1]), sl2, -m));
              rs4[i & 3] += x0 + x1;
              pk[i] = pack_bf16x2(x0, x1);
            }
            tm_st32(s_lane + 32 * half, pk);
          }
          return (rs4[0] + rs4[1]) + (rs4[2] + rs4[3]);
        };
        // Exact tile max; raise m where it exceeds m + kRescale (rescaling O).
        auto raise_to_max = [&]() {
          float mx8[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) mx8[i] = __uint_as_float(v[i]);
#pragma unroll
          for (int i = 8; i < KT; ++i) mx8[i & 7] = fmaxf(mx8[i & 7], __uint_as_float(v[i]));
          float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                           fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
          mx *= sl2;
          const bool raise = mx > m + kRescale;
          if (__any_sync(0xffffffffu, raise)) {
            const float m_new = raise ? mx : m;
            const float a = ex2_approx_ftz(m - m_new);
            l *= a;
            m = m_new;
            if (j > 0) {
#pragma unroll 1
              for (int c = 0; c < HD; c += 32) {
                uint32_t o[32];
                tm_ld32(o_lane + c, o);
#pragma unroll
                for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * a);
                tm_st32(o_lane + c, o);
              }
            }
          }
        };
        float rs;
        if (j == 0) {
          raise_to_max();
          rs = exp_tile();
        } else {
          // Against m without this tile's max; redone with it only when a row's
          // sum would pass kSumLimit.
          rs = exp_tile();
          if (__any_sync(0xffffffffu, !(rs <= kSumLimit))) {
            raise_to_max();
            rs = exp_tile();
          }
        }
        l += rs;
        tm_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&pfull[g]);
      }
      if (!ok) break;
      // Output: the item's last PV_g done; O_g / l to bf16, straight to global
      // memory (this thread's row), then O_g handed back for the next item.
      ok = mbar_wait(&odone[g], it & 1, abort_flag, err, CORA_DERR_EPI_WAIT);
      if (!ok) break;
      tc_fence_after();
      const int qrow = (pr * 2 + g) * QT + r;  // relative to q_start
      const bool store = qrow < q_len;
      uint16_t* orow = out + (static_cast<int64_t>(b) * q_len + qrow) * ldo + h * HD;
      const float inv = 1.f / l;
#pragma unroll 1
      for (int c = 0; c < HD; c += 32) {
        uint32_t o[32];
        tm_ld32(o_lane + c, o);
        if (store) {
#pragma unroll
          for (int i = 0; i < 32; i += 8) {
            const uint4 w = make_uint4(pack_bf16x2(__uint_as_float(o[i]) * inv, __uint_as_float(o[i + 1]) * inv),
                                       pack_bf16x2(__uint_as_float(o[i + 2]) * inv, __uint_as_float(o[i + 3]) * inv),
                                       pack_bf16x2(__uint_as_float(o[i + 4]) * inv, __uint_as_float(o[i + 5]) * inv),
                                       pack_bf16x2(__uint_as_float(o[i + 6]) * inv, __uint_as_float(o[i + 7]) * inv));
            *reinterpret_cast<uint4*>(orow + c + i) = w;
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&oempty[g]);
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

cudaError_t attention_tc2_prepare() {
  return cudaFuncSetAttribute(attention_tc2_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, attn2::SMEM);
}

cudaError_t launch_attention_tc2(const CUtensorMap& tmQKV, uint16_t* out, int B, int S, int Hq, int Hkv, int q_start,
                                 int q_len, int* err, int num_sms, cudaStream_t st) {
  const int n_qt = (q_len + attn2::QT - 1) / attn2::QT;
  const int n_pairs = (n_qt + 1) / 2;
  const int n_items = n_pairs * Hq * B;
  const int grid = n_items < num_sms ? n_items : num_sms;
  return launch_pdl(attention_tc2_kernel, dim3(grid), dim3(attn2::THREADS), attn2::SMEM, st, tmQKV, out, S, Hq, Hkv,
                    q_start, q_len, n_pairs, n_items, err);
}
