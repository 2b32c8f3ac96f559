// Offline similarity on the tensor cores (Section III-B, Eqs. 3-5; Alg. 1)
// for E in {8, 16, 32, 64}:
//   sim_logits_kernel<E>: H = X_cal W^T for the L routers stacked (W rows =
//     L * E), one 128-token x 256-logit tile per step of a persistent loop
//     (TMA ring, tcgen05.mma, two TMEM accumulators, as in the expert FFN).
//     The epilogue writes H in fp32, token-major (the workspace contract),
//     writes H^T as two bf16 planes, hi = bf16(h) and lo = bf16(h - hi),
//     expert-major so that the Gram reads both K-major, and counts each
//     token's top-k_freq experts of every layer (Eq. 5) in a shared-memory
//     histogram.
//   gram_tc_kernel: partial Grams of 64 consecutive rows of H^T (64 / E
//     layers) over a range of tokens. The 64 hi rows and the same 64 lo rows
//     form one 128-row tile A, and one tcgen05 MMA per K step accumulates
//     A A^T, whose four 64 x 64 quadrants are hi hi^T, hi lo^T, lo hi^T and
//     lo lo^T: the epilogue adds them, (hi hi^T + hi lo^T) + (lo hi^T +
//     lo lo^T) = (hi + lo)(hi + lo)^T in fp32, and keeps the diagonal blocks
//     (rows and columns of the same layer: Eq. 4's inner products). The
//     partials are then reduced in fp64 in a fixed order.
// Every wait is bounded; a wait that runs out reports ORDERMOE_DEV_WAIT_TIMEOUT,
// stops the other roles, drains the copies and MMAs in flight and returns.
#include <mutex>

#include "common.cuh"

namespace om {

namespace gg {
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_fn();
}  // namespace gg

static __device__ unsigned long long g_err_simtc = 0;

int read_clear_err_simtc(unsigned long long* out) {
  unsigned long long zero = 0;
  OM_CUDA(cudaMemcpyFromSymbol(out, g_err_simtc, sizeof(*out)));
  OM_CUDA(cudaMemcpyToSymbol(g_err_simtc, &zero, sizeof(zero)));
  return ORDERMOE_OK;
}

namespace sg {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;  // bf16 elements = one 128-byte swizzled row
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int BOX_BYTES = 128 * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + 2 * BOX_BYTES;
constexpr int THREADS = 192;    // Gram: TMA, MMA, 4 epilogue warps
constexpr int L_EPI_WARPS = 16;  // logits epilogue: four warps per TMEM lane quarter
constexpr int L_THREADS = 64 + 32 * L_EPI_WARPS;  // + TMA and MMA warps
constexpr int TMEM_COLS = 512;
constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN);
constexpr int MAX_HIST = 4096;  // L * E counters in shared memory

constexpr int G_ROWS = 64;  // rows of H^T per Gram block
constexpr int G_BOX_BYTES = G_ROWS * BK * 2;
constexpr int G_STAGES = 12;
constexpr int G_STAGE_BYTES = 2 * G_BOX_BYTES;  // hi and lo boxes, 64 rows x 64 tokens each
constexpr int G_TMEM_COLS = 128;
constexpr uint32_t G_IDESC = idesc_bf16_f32(128, 128);

// CTA-pair variant of the logits kernel: a pair computes 256 tokens x 256
// columns with one cta_group::2 MMA (M = 256 across the pair, each CTA's
// TMEM holding its 128 tokens); each CTA loads its 128 tokens and half of the
// 256 weight rows per K step (32 KB instead of 48 KB: a third less L2 -> shared
// memory traffic per flop), six stages deep.
constexpr int P_STAGES = 6;
constexpr int P_STAGE_BYTES = A_BYTES + BOX_BYTES;
constexpr int L_MAX_STAGES = P_STAGES > STAGES ? P_STAGES : STAGES;
static_assert(P_STAGES * P_STAGE_BYTES <= STAGES * STAGE_BYTES, "pair ring fits the 1-CTA ring's space");

struct LSmem {
  uint64_t full[L_MAX_STAGES];
  uint64_t empty[L_MAX_STAGES];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
  int zero;
};
constexpr int L_SMEM_FIXED = STAGES * STAGE_BYTES + 1024 + static_cast<int>(sizeof(LSmem));

struct GSmem {
  uint64_t full[G_STAGES];
  uint64_t empty[G_STAGES];
  uint64_t tfull;
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
  int zero;
};
constexpr int G_SMEM_BYTES = G_STAGES * G_STAGE_BYTES + 1024 + static_cast<int>(sizeof(GSmem));

struct LArgs {
  int N;            // calibration tokens (rows of X)
  int C;            // L * E logit columns
  int K;            // d
  int n_tiles;      // 256-column slices
  int L;
  int kf;           // k_freq of Eq. 5
  float* H;         // [N][C] fp32, or null: not written
  uint16_t* hi;     // [C][ldT] bf16
  uint16_t* lo;     // [C][ldT] bf16
  int ldT;
  int32_t* counts;  // [C] (added to)
  uint64_t limit_ns;
};

struct GArgs {
  int R;            // L * E rows of H^T
  int E;
  int kblocks;      // 64-token steps over all tokens
  int kb_per_split;
  int nsplit;
  float* gpart;     // [L][nsplit][64][64]
  uint64_t limit_ns;
};

// larger logit first, equal logits by lower index (the rank order of Eq. 5's
// top-k): each pass keeps the first unused maximum (strict >, from -inf), so
// finite logits rank exactly as that order says.
template <int E>
__device__ __forceinline__ void count_topk(const float (&x)[E], int kf, int* hist_row) {
  unsigned long long used = 0;
  for (int j = 0; j < kf; ++j) {
    int best = -1;
    float bv = -INFINITY;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const bool take = !(used & (1ull << e)) && x[e] > bv;
      best = take ? e : best;
      bv = take ? x[e] : bv;
    }
    if (best < 0) return;
    used |= 1ull << best;
    atomicAdd(&hist_row[best], 1);
  }
}

// The top-k_freq set of 64 logits as a bit mask (experts 0-31 in lo, 32-63
// in hi), by the rules of count_topk.
__device__ __forceinline__ void topk_mask64_passes(const float (&x)[64], int kf, uint32_t& lo,
                                                   uint32_t& hi) {
  unsigned long long used = 0;
  for (int j = 0; j < kf; ++j) {
    int best = -1;
    float bv = -INFINITY;
#pragma unroll
    for (int e = 0; e < 64; ++e) {
      const bool take = !(used & (1ull << e)) && x[e] > bv;
      best = take ? e : best;
      bv = take ? x[e] : bv;
    }
    if (best < 0) break;
    used |= 1ull << best;
  }
  lo = static_cast<uint32_t>(used);
  hi = static_cast<uint32_t>(used >> 32);
}

// 32 x 32 bit transpose across a warp: lane r holds row r (bit c = entry
// (r, c)); afterwards lane c holds column c (bit r = entry (r, c)). Each step
// swaps the off-diagonal s x s blocks of every 2s x 2s block between lanes r
// and r ^ s.
__device__ __forceinline__ uint32_t warp_transpose32(uint32_t x, int lane) {
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) {
    const uint32_t keep = s == 16 ? 0x0000FFFFu : s == 8 ? 0x00FF00FFu : s == 4 ? 0x0F0F0F0Fu
                          : s == 2 ? 0x33333333u : 0x55555555u;  // columns with bit s clear
    const uint32_t y = __shfl_xor_sync(0xffffffffu, x, s);
    x = (lane & s) ? ((x & ~keep) | ((y & ~keep) >> s)) : ((x & keep) | ((y & keep) << s));
  }
  return x;
}

// NK: 6 or 8 = Eq. 5's counts of 64-expert layers with a network keeping the
// NK largest logits (k_freq <= NK), streamed over the two 32-logit halves of
// a layer; 0 = the selection passes over all 64 (k_freq > 8) or E < 64.
// PAIR: clusters of two CTAs with cta_group::2 MMAs (see P_STAGES).
template <int E, int NK, bool PAIR>
__global__ void __launch_bounds__(L_THREADS, 1)
    sim_logits_kernel(const __grid_constant__ CUtensorMap mapX, const __grid_constant__ CUtensorMap mapW,
                      LArgs args) {
  constexpr int KSTAGES = PAIR ? P_STAGES : STAGES;
  constexpr int KSTAGE_BYTES = PAIR ? P_STAGE_BYTES : STAGE_BYTES;
  constexpr int TBM = PAIR ? 2 * BM : BM;  // tokens per tile
  extern __shared__ uint8_t smem_raw[];
  uint8_t* tiles = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  LSmem& s = *reinterpret_cast<LSmem*>(tiles + STAGES * STAGE_BYTES);
  int* hist = reinterpret_cast<int*>(tiles + STAGES * STAGE_BYTES + sizeof(LSmem));
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const uint32_t rp = PAIR ? (cluster_ctarank() & 1u) : 0u;  // rank within the pair
  const int cid = PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int ncl = PAIR ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);
  for (int i = tid; i < args.C; i += blockDim.x) hist[i] = 0;
  if (tid == 0) {
    for (int i = 0; i < KSTAGES; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.tfull[i], 1);
      // pair: one arrive per epilogue warp of either CTA, on the even CTA's barrier
      mbar_init(&s.tempty[i], PAIR ? 2 * L_EPI_WARPS : 32 * L_EPI_WARPS);
    }
    mbar_init(&s.drain, 1);
    s.abort = 0;
    s.zero = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&mapX);
    tma_prefetch_map(&mapW);
  }
  if (warp == 1) {
    if (PAIR) {
      tmem_alloc_pair(&s.tmem_base, TMEM_COLS);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(&s.tmem_base, TMEM_COLS);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  if (PAIR) cluster_sync();  // barriers of both CTAs initialised, TMEM allocated
  else __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = s.tmem_base;
  const int total = ((args.N + TBM - 1) / TBM) * args.n_tiles;
  const int kblocks = args.K / BK;
  volatile int* abort = &s.abort;
  uint32_t issued_mask = 0, last_phase_bits = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (int tile = cid; tile < total && !*abort; tile += ncl) {
        const int mt = tile / args.n_tiles, n = tile - mt * args.n_tiles;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&s.empty[stage], phase ^ 1u, args.limit_ns, abort)) {
            if (!*abort) report(&g_err_simtc, ORDERMOE_DEV_WAIT_TIMEOUT, 11);
            *abort = 1;
            break;
          }
          uint8_t* sa = tiles + stage * KSTAGE_BYTES;
          if (PAIR) {
            // this CTA's 128 tokens and 128 of the tile's 256 weight rows; both
            // CTAs' bytes complete on the even CTA's barrier
            const uint32_t full_even = mapa_shared(smem_u32(&s.full[stage]), 0);
            if (rp == 0) mbar_arrive_expect_tx(&s.full[stage], 2 * P_STAGE_BYTES);
            tma_load_2d_pair(sa, &mapX, full_even, kb * BK, mt * TBM + static_cast<int>(rp) * BM);
            tma_load_2d_pair(sa + A_BYTES, &mapW, full_even, kb * BK, n * BN + static_cast<int>(rp) * 128);
          } else {
            mbar_arrive_expect_tx(&s.full[stage], STAGE_BYTES);
            tma_load_2d(sa, &mapX, &s.full[stage], kb * BK, mt * BM);
            tma_load_2d(sa + A_BYTES, &mapW, &s.full[stage], kb * BK, n * BN);
            tma_load_2d(sa + A_BYTES + BOX_BYTES, &mapW, &s.full[stage], kb * BK, n * BN + 128);
          }
          issued_mask |= 1u << stage;
          last_phase_bits = (last_phase_bits & ~(1u << stage)) | (phase << stage);
          if (++stage == KSTAGES) { stage = 0; phase ^= 1u; }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rp == 0) {  // pair: the even CTA issues the pair's MMAs
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int tile = cid; tile < total && !*abort; tile += ncl, ++it) {
        const int slot = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait(&s.tempty[slot], acc_phase ^ 1u, args.limit_ns, abort)) {
          if (!*abort) report(&g_err_simtc, ORDERMOE_DEV_WAIT_TIMEOUT, 12);
          *abort = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + slot * BN;
        bool ok = true;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&s.full[stage], phase, args.limit_ns, abort)) {
            if (!*abort) report(&g_err_simtc, ORDERMOE_DEV_WAIT_TIMEOUT, 13);
            *abort = 1;
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(tiles + stage * KSTAGE_BYTES);
          const uint32_t b0 = a0 + A_BYTES;
          if (PAIR) {
            constexpr uint32_t PIDESC = idesc_bf16_f32(256, BN);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
              mma_bf16_pair(d_tmem, sdesc_kmajor_sw128(a0 + kk * 32),
                            sdesc_kmajor_sw128(b0 + kk * 32), PIDESC, (kb | kk) != 0 ? 1u : 0u);
            mma_issued = true;
            mma_commit_pair(&s.empty[stage], 0x3);
          } else {
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
              mma_bf16(d_tmem, sdesc_kmajor_sw128(a0 + kk * 32), sdesc_kmajor_sw128(b0 + kk * 32),
                       IDESC, (kb | kk) != 0 ? 1u : 0u);
            mma_issued = true;
            mma_commit(&s.empty[stage]);
          }
          if (++stage == KSTAGES) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        if (PAIR) mma_commit_pair(&s.tfull[slot], 0x3);
        else mma_commit(&s.tfull[slot]);
      }
    }
  } else {
    // epilogue: warps 2..17; warp w reads TMEM lane quarter w % 4 (thread = one
    // token) and the 64-column quarter (w - 2) / 4 of the tile
    const int q = warp & 3;
    const int part = (warp - 2) >> 2;
    const int lrow = q * 32 + lane;
    int it = 0;
    for (int tile = cid; tile < total; tile += ncl, ++it) {
      if (__any_sync(0xffffffffu, *abort != 0)) break;
      const int slot = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&s.tfull[slot], acc_phase, args.limit_ns, abort));
      if (!ok) {
        if (lane == 0 && !*abort) report(&g_err_simtc, ORDERMOE_DEV_WAIT_TIMEOUT, 14);
        *abort = 1;
        break;
      }
      tc_fence_after();
      const int mt = tile / args.n_tiles, n = tile - mt * args.n_tiles;
      const int row = mt * TBM + static_cast<int>(rp) * BM + lrow;
      const bool valid = row < args.N;
      const uint32_t tb = tmem_base + slot * BN + (static_cast<uint32_t>(q * 32) << 16);
      float* orow = args.H + (size_t)row * args.C;
      float prev[32];  // E == 64, NK == 0: the first half of a layer's logits
      float net[NK > 0 ? NK : 1];  // E == 64, NK > 0: the NK largest logits so far, descending
#pragma unroll
      for (int half = 0; half < 2; ++half) {  // the two 32-column chunks of the warp's part
        const int c = 2 * part + half;
        const int cb = n * BN + c * 32;
        if (cb >= args.C) break;  // warp-uniform
        uint32_t v[32];
        tmem_ld32(tb + c * 32, v);
        tmem_ld_wait();
        const int nv = min(32, args.C - cb);  // C is a multiple of 8, so nv is even
        // hi/lo planes: each lane converts two adjacent logits at a time, and
        // the lanes of a pair (tokens 2k, 2k + 1) swap halves so that the even
        // lane holds expert i and the odd lane expert i + 1 of both tokens:
        // one 4-byte store per plane and expert pair (ldT and the even row
        // keep it aligned; row 2k + 1 < ldT whenever row 2k < N)
        {
          const int odd = lane & 1;
          const uint32_t psel = odd ? 0x3276u : 0x5410u;
          const size_t orow_pair = static_cast<size_t>(row & ~1) + (size_t)(cb + odd) * args.ldT;
          const bool pair_valid = (row & ~1) < args.N;
#pragma unroll
          for (int i = 0; i < 32; i += 2) {
            if (i >= nv) break;  // warp-uniform
            const float2 x2 = make_float2(__uint_as_float(v[i]), __uint_as_float(v[i + 1]));
            const __nv_bfloat162 h2 = __float22bfloat162_rn(x2);
            // x - hi, exact: one packed fma with -1
            const float2 r2 = __ffma2_rn(__bfloat1622float2(h2), make_float2(-1.0f, -1.0f), x2);
            const __nv_bfloat162 l2 = __float22bfloat162_rn(r2);
            const uint32_t hw = *reinterpret_cast<const uint32_t*>(&h2);
            const uint32_t lw = *reinterpret_cast<const uint32_t*>(&l2);
            const uint32_t hp = __shfl_xor_sync(0xffffffffu, hw, 1);
            const uint32_t lp = __shfl_xor_sync(0xffffffffu, lw, 1);
            if (pair_valid) {
              const size_t o = orow_pair + (size_t)i * args.ldT;
              *reinterpret_cast<uint32_t*>(args.hi + o) = __byte_perm(hw, hp, psel);
              *reinterpret_cast<uint32_t*>(args.lo + o) = __byte_perm(lw, lp, psel);
            }
          }
        }
        if (valid && args.H != nullptr) {  // logits kept only when asked for
          float4* dst = reinterpret_cast<float4*>(orow + cb);
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (4 * i < nv)
              dst[i] = make_float4(__uint_as_float(v[4 * i]), __uint_as_float(v[4 * i + 1]),
                                   __uint_as_float(v[4 * i + 2]), __uint_as_float(v[4 * i + 3]));
        }
        if (E == 64 && NK > 0) {
          // Eq. 5 for one layer and the warp's 32 tokens with fewer
          // compare/select operations than the passes: a descending min/max
          // insertion network keeps the NK largest logits with multiplicity
          // (min(v[j-1], max(v[j], x)) in slot j leaves v as it was for a NaN
          // x), T = the k_freq-th of them, and every logit >= T is selected;
          // when more than k_freq logits reach T (equal logits at the
          // boundary), the surplus equal to T is taken back from the highest
          // index down, which leaves the lowest indices, as the rank order
          // says; -inf logits are never selected, as in the passes. The
          // network takes the layer's first 32 logits (each lane's token),
          // then the next 32; with T known the first half is read from TMEM
          // again for its mask. Each lane's top-k set becomes a 64-bit mask,
          // the masks are transposed across the warp, and lane j adds the
          // number of tokens that select expert j (and j + 32): two
          // conflict-free shared-memory adds per lane.
          if (half == 0) {
#pragma unroll
            for (int i = 0; i < NK; ++i) net[i] = -INFINITY;
          }
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float x = __uint_as_float(v[i]);
#pragma unroll
            for (int j = NK - 1; j > 0; --j) net[j] = fminf(net[j - 1], fmaxf(net[j], x));
            net[0] = fmaxf(net[0], x);
          }
          if (half == 1) {
            // T = net[kf - 1], the smallest of the first kf (net is descending),
            // written as a running minimum so that net stays in registers
            float T = net[0];
#pragma unroll
            for (int j = 1; j < NK; ++j) T = j < args.kf ? fminf(T, net[j]) : T;
            const float Tc = fmaxf(T, -3.402823466e38f);  // below every finite logit, above -inf
            uint32_t mhi = 0u, ehi = 0u, mlo = 0u, elo = 0u;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float x = __uint_as_float(v[i]);
              mhi |= x >= Tc ? (1u << i) : 0u;
              ehi |= x == T ? (1u << i) : 0u;
            }
            tmem_ld32(tb + (c - 1) * 32, v);  // the first half again
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float x = __uint_as_float(v[i]);
              mlo |= x >= Tc ? (1u << i) : 0u;
              elo |= x == T ? (1u << i) : 0u;
            }
            unsigned long long sel = valid ? ((static_cast<unsigned long long>(mhi) << 32) | mlo) : 0ull;
            const unsigned long long eq = (static_cast<unsigned long long>(ehi) << 32) | elo;
            // equal logits straddling the boundary: take back the surplus from the highest index
            for (int extra = __popcll(sel) - args.kf; extra > 0 && (sel & eq) != 0ull; --extra)
              sel &= ~(1ull << (63 - __clzll(sel & eq)));
            const int l = (cb - 32) / 64;
            const int nlo = __popc(warp_transpose32(static_cast<uint32_t>(sel), lane));
            const int nhi = __popc(warp_transpose32(static_cast<uint32_t>(sel >> 32), lane));
            if (nlo) atomicAdd(&hist[l * 64 + lane], nlo);
            if (nhi) atomicAdd(&hist[l * 64 + 32 + lane], nhi);
          }
        } else if (E == 64) {
          // k_freq > 8: the selection passes over the layer's 64 logits
          if ((c & 1) == 0) {
#pragma unroll
            for (int i = 0; i < 32; ++i) prev[i] = __uint_as_float(v[i]);
          } else {
            uint32_t mlo = 0u, mhi = 0u;
            if (valid) {
              float x[64];
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                x[i] = prev[i];
                x[32 + i] = __uint_as_float(v[i]);
              }
              topk_mask64_passes(x, args.kf, mlo, mhi);
            }
            const int l = (cb - 32) / 64;
            const int nlo = __popc(warp_transpose32(mlo, lane));
            const int nhi = __popc(warp_transpose32(mhi, lane));
            if (nlo) atomicAdd(&hist[l * 64 + lane], nlo);
            if (nhi) atomicAdd(&hist[l * 64 + 32 + lane], nhi);
          }
        } else if (valid) {
#pragma unroll
          for (int sub = 0; sub < 32 / E; ++sub) {
            float x[E];
#pragma unroll
            for (int i = 0; i < E; ++i) x[i] = __uint_as_float(v[sub * E + i]);
            const int l = (cb + sub * E) / E;
            if (l < args.L) count_topk<E>(x, args.kf, hist + l * E);
          }
        }
      }
      tc_fence_before();
      if (PAIR) {
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(mapa_shared(smem_u32(&s.tempty[slot]), 0));
      } else {
        mbar_arrive(&s.tempty[slot]);
      }
    }
  }

  __syncthreads();
  if (s.abort) {
    // drain the copies (pair: all complete on the even CTA's barriers) and
    // the MMAs in flight, both bounded
    volatile int* never = &s.zero;
    if (warp == 0 && lane == 0 && rp == 0) {
      for (int st = 0; st < KSTAGES; ++st)
        if ((issued_mask >> st) & 1u)
          mbar_wait(&s.full[st], (last_phase_bits >> st) & 1u, args.limit_ns, never);
    }
    if (warp == 1 && lane == 0 && rp == 0 && mma_issued) {
      if (PAIR) mma_commit_pair(&s.drain, 0x1);
      else mma_commit(&s.drain);
      mbar_wait(&s.drain, 0, args.limit_ns, never);
    }
    __syncthreads();
  }
  if (PAIR) {
    tc_fence_before();
    cluster_sync();  // both CTAs done: no more arrivals or copies into either
    tc_fence_after();
  }
  for (int i = tid; i < args.C; i += blockDim.x)
    if (hist[i]) atomicAdd(&args.counts[i], hist[i]);
  if (warp == 1) {
    tc_fence_after();
    if (PAIR) tmem_dealloc_pair(tmem_base, TMEM_COLS);
    else tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// The AND of v over the 128 epilogue threads (warps 2..5, named barrier 1),
// returned to all of them: a barrier that every epilogue thread reaches.
__device__ __forceinline__ bool epi_and(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, 1, 128, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(v))
      : "memory");
  return r != 0;
}

// grid (row blocks of 64 rows of H^T, token splits)
__global__ void __launch_bounds__(THREADS, 1)
    gram_tc_kernel(const __grid_constant__ CUtensorMap mapHi, const __grid_constant__ CUtensorMap mapLo,
                   GArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* tiles = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  GSmem& s = *reinterpret_cast<GSmem*>(tiles + G_STAGES * G_STAGE_BYTES);
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int rb = blockIdx.x, split = blockIdx.y;
  const int kb0 = split * args.kb_per_split;
  const int kb1 = min(kb0 + args.kb_per_split, args.kblocks);
  const int nkb = kb1 > kb0 ? kb1 - kb0 : 0;
  if (tid == 0) {
    for (int i = 0; i < G_STAGES; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 1);
    }
    mbar_init(&s.tfull, 1);
    mbar_init(&s.drain, 1);
    s.abort = 0;
    s.zero = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&mapHi);
    tma_prefetch_map(&mapLo);
  }
  if (warp == 1) {
    tmem_alloc(&s.tmem_base, G_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = s.tmem_base;
  volatile int* abort = &s.abort;
  uint32_t issued_mask = 0, last_phase_bits = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (int i = 0; i < nkb && !*abort; ++i) {
        if (!mbar_wait(&s.empty[stage], phase ^ 1u, args.limit_ns, abort)) {
          if (!*abort) report(&g_err_simtc, ORDERMOE_DEV_WAIT_TIMEOUT, 21);
          *abort = 1;
          break;
        }
        uint8_t* st = tiles + stage * G_STAGE_BYTES;
        mbar_arrive_expect_tx(&s.full[stage], G_STAGE_BYTES);
        tma_load_2d(st, &mapHi, &s.full[stage], (kb0 + i) * BK, rb * G_ROWS);
        tma_load_2d(st + G_BOX_BYTES, &mapLo, &s.full[stage], (kb0 + i) * BK, rb * G_ROWS);
        issued_mask |= 1u << stage;
        last_phase_bits = (last_phase_bits & ~(1u << stage)) | (phase << stage);
        if (++stage == G_STAGES) { stage = 0; phase ^= 1u; }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && nkb > 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int i = 0; i < nkb; ++i) {
        if (!mbar_wait(&s.full[stage], phase, args.limit_ns, abort)) {
          if (!*abort) report(&g_err_simtc, ORDERMOE_DEV_WAIT_TIMEOUT, 22);
          *abort = 1;
          ok = false;
          break;
        }
        tc_fence_after();
        // A = [hi; lo] (128 rows, the two boxes back to back), D += A A^T
        const uint32_t a0 = smem_u32(tiles + stage * G_STAGE_BYTES);
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          const uint64_t da = sdesc_kmajor_sw128(a0 + kk * 32);
          mma_bf16(tmem_base, da, da, G_IDESC, (i | kk) != 0 ? 1u : 0u);
        }
        mma_issued = true;
        mma_commit(&s.empty[stage]);
        if (++stage == G_STAGES) { stage = 0; phase ^= 1u; }
      }
      if (ok) mma_commit(&s.tfull);
    }
  } else {
    // epilogue: warp q reads TMEM lanes 32 q .. 32 q + 31: rows 0..63 of D
    // are the hi rows, 64..127 the lo rows of the block's 64 rows of H^T.
    // Each thread adds its row's two column halves (x hi^T + x lo^T); the lo
    // threads hand theirs over through shared memory (the consumed ring) and
    // the hi threads add them: G = (hi hi^T + hi lo^T) + (lo hi^T + lo lo^T).
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const int i = r & (G_ROWS - 1);  // row of the block
    const int gr = rb * G_ROWS + i;  // row of H^T
    const int E = args.E;
    const int l = gr / E, ii = gr - l * E;
    const int c0 = l * E - rb * G_ROWS;  // the layer's first column in the block
    float* xch = reinterpret_cast<float*>(tiles);  // [64][65] lo-row sums
    bool ok = true;
    if (nkb > 0) {
      ok = __all_sync(0xffffffffu, mbar_wait(&s.tfull, 0, args.limit_ns, abort));
      if (!ok && lane == 0 && !*abort) report(&g_err_simtc, ORDERMOE_DEV_WAIT_TIMEOUT, 23);
      if (!ok) *abort = 1;
    }
    // the same decision in all four epilogue warps (they meet at a barrier below)
    const bool go = epi_and(ok && *abort == 0);
    if (go) {
      tc_fence_after();
      // the layer's columns: E == 64 -> both 32-column chunks of each half;
      // E <= 32 -> the chunk q & 1 only (a warp's 32 rows and their layers'
      // columns lie in the same aligned 32-row range), warp-uniform either way
      float sum[64];
#pragma unroll
      for (int x = 0; x < 64; ++x) sum[x] = 0.0f;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (E < 64 && h != (q & 1)) continue;
        uint32_t v0[32], v1[32];
        if (nkb > 0) {
          tmem_ld32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + h * 32, v0);
          tmem_ld32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + 64 + h * 32, v1);
          tmem_ld_wait();
#pragma unroll
          for (int x = 0; x < 32; ++x)
            sum[h * 32 + x] = __fadd_rn(__uint_as_float(v0[x]), __uint_as_float(v1[x]));
        }
      }
      if (r >= G_ROWS) {
#pragma unroll
        for (int x = 0; x < 64; ++x) xch[i * 65 + x] = sum[x];
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (r < G_ROWS && gr < args.R) {
        float* dst = args.gpart + (((size_t)l * args.nsplit + split) * 64 + ii) * 64;
#pragma unroll
        for (int x = 0; x < 64; ++x)
          if (x >= c0 && x < c0 + E) dst[x - c0] = __fadd_rn(sum[x], xch[i * 65 + x]);
      }
    }
  }

  __syncthreads();
  if (s.abort) {
    volatile int* never = &s.zero;
    if (warp == 0 && lane == 0) {
      for (int st = 0; st < G_STAGES; ++st)
        if ((issued_mask >> st) & 1u)
          mbar_wait(&s.full[st], (last_phase_bits >> st) & 1u, args.limit_ns, never);
    }
    if (warp == 1 && lane == 0 && mma_issued) {
      mma_commit(&s.drain);
      mbar_wait(&s.drain, 0, args.limit_ns, never);
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, G_TMEM_COLS);
  }
}

// 2-D bf16 map over [rows][cols] with row pitch ld elements (ld * 2 a multiple
// of 16 bytes), a 64-column x 64-row box (the Gram's) and the 128-byte
// swizzle; reads past cols or rows return zeros.
int make_map_ld(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld) {
  gg::EncodeTiledFn enc = gg::encode_fn();
  if (!enc) return fail(ORDERMOE_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {BK, G_ROWS};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(ORDERMOE_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return ORDERMOE_OK;
}

}  // namespace sg

bool sim_tc_supported(int L, int E) {
  return (E == 8 || E == 16 || E == 32 || E == 64) && (long long)L * E <= sg::MAX_HIST;
}

// Layers per block of the pipelined plan: 512 logit columns (four 128-row
// blocks of H^T for the Gram). Every block streams all of X_cal once; with
// 512 columns a block's GEMM stays compute-bound (about 410 flops per byte).
int sim_tc_part_layers(int E) { return E >= 512 ? 1 : 512 / E; }

// Most token splits of the Gram (the workspace holds this many partials).
int sim_tc_max_splits() { return 256; }

// Token splits of the Gram. They depend on E and N only (the row blocks of
// one part of the pipelined plan fill the GPU), so the partial sums, and the
// similarities, are the same whether the layers are done in one call or part
// by part.
int sim_tc_nsplit(int L, int E, int64_t N) {
  const int part = sim_tc_part_layers(E);
  const int n_rb = ((L < part ? L : part) * E + sg::G_ROWS - 1) / sg::G_ROWS;
  const int kblocks = static_cast<int>((N + sg::BK - 1) / sg::BK);
  const int sms = num_sms() > 1 ? num_sms() - 1 : 1;  // the pipelined plan keeps one SM free
  int ns = sms / n_rb;
  if (ns < 1) ns = 1;
  if (ns > kblocks) ns = kblocks;
  if (ns > sim_tc_max_splits()) ns = sim_tc_max_splits();
  return ns;
}

// Largest dynamic shared memory a block may ask for: asking for it keeps any
// other kernel's block off that SM.
static int whole_sm_smem() {
  int dev = 0, v = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
    return 0;
  return v;
}

// H [N][L E] fp32, the hi/lo planes [L E][ldT], counts (zeroed by the caller),
// and the partial Grams gpart [L][nsplit][64][64]. reserve_sm: run on all SMs
// but one and take each SM's whole shared memory, so that the one left over
// takes the kernels of another stream (the pipelined plan's grouping and
// placement) without slowing a block of these persistent grids.
int sim_tc_launch(const uint16_t* X, int N, const uint16_t* W, int L, int E, int d, int kf,
                  float* H, uint16_t* hi, uint16_t* lo, int ldT, int32_t* counts, float* gpart,
                  int nsplit, bool reserve_sm, cudaStream_t stream) {
  using namespace sg;
  const int C = L * E;
  size_t lsmem = L_SMEM_FIXED + sizeof(int) * (size_t)C;
  size_t gsmem = G_SMEM_BYTES;
  static PerDevice cache;
  const cudaError_t attr_err = static_cast<cudaError_t>(per_device(cache, [] {
    int lmax = L_SMEM_FIXED + static_cast<int>(sizeof(int)) * MAX_HIST;
    int gmax = G_SMEM_BYTES;
    const int whole = whole_sm_smem();
    if (whole > lmax) lmax = whole;
    if (whole > gmax) gmax = whole;
    cudaError_t e = cudaFuncSetAttribute(sim_logits_kernel<8, 0, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, lmax);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(sim_logits_kernel<16, 0, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, lmax);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(sim_logits_kernel<32, 0, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, lmax);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(sim_logits_kernel<64, 6, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, lmax);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(sim_logits_kernel<64, 8, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, lmax);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(sim_logits_kernel<64, 0, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, lmax);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(gram_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, gmax);
    return static_cast<int>(e);
  }));
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(similarity)");
  CUtensorMap mX, mW, mHi, mLo;
  int rc;
  if ((rc = make_tmap_bf16(&mX, X, N, d, 128))) return rc;
  if ((rc = make_tmap_bf16(&mW, W, C, d, 128))) return rc;
  if ((rc = make_map_ld(&mHi, hi, C, N, ldT))) return rc;
  if ((rc = make_map_ld(&mLo, lo, C, N, ldT))) return rc;
  LArgs la{};
  la.N = N;
  la.C = C;
  la.K = d;
  la.n_tiles = (C + BN - 1) / BN;
  la.L = L;
  la.kf = kf;
  la.H = H;
  la.hi = hi;
  la.lo = lo;
  la.ldT = ldT;
  la.counts = counts;
  la.limit_ns = wait_limit_ns();
  const long long tiles = (long long)((N + BM - 1) / BM) * la.n_tiles;
  int sms = num_sms();
  if (reserve_sm && sms > 1) {
    --sms;
    const size_t whole = static_cast<size_t>(whole_sm_smem());
    if (whole > lsmem) lsmem = whole;
    if (whole > gsmem) gsmem = whole;
  }
  const int grid = static_cast<int>(tiles < sms ? tiles : sms);
  if (E == 64 && kf <= 8) {
    // CTA pairs over 256-token tiles, at most one pair per two SMs
    const long long ptiles = (long long)((N + 2 * BM - 1) / (2 * BM)) * la.n_tiles;
    const int pairs = static_cast<int>(ptiles < sms / 2 ? ptiles : sms / 2);
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr;
    cfg.gridDim = dim3(2 * (pairs > 0 ? pairs : 1), 1, 1);
    cfg.blockDim = dim3(L_THREADS, 1, 1);
    cfg.dynamicSmemBytes = lsmem;
    cfg.stream = stream;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 2;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    const cudaError_t e = kf <= 6 ? cudaLaunchKernelEx(&cfg, sim_logits_kernel<64, 6, true>, mX, mW, la)
                                  : cudaLaunchKernelEx(&cfg, sim_logits_kernel<64, 8, true>, mX, mW, la);
    if (e != cudaSuccess) return cuda_fail(e, "sim_logits_kernel (CTA pairs)");
  } else {
    switch (E) {
      case 8: sim_logits_kernel<8, 0, false><<<grid, L_THREADS, lsmem, stream>>>(mX, mW, la); break;
      case 16: sim_logits_kernel<16, 0, false><<<grid, L_THREADS, lsmem, stream>>>(mX, mW, la); break;
      case 32: sim_logits_kernel<32, 0, false><<<grid, L_THREADS, lsmem, stream>>>(mX, mW, la); break;
      default: sim_logits_kernel<64, 0, false><<<grid, L_THREADS, lsmem, stream>>>(mX, mW, la); break;
    }
  }
  OM_LAUNCHED("sim_logits_kernel");
  GArgs ga{};
  ga.R = C;
  ga.E = E;
  ga.kblocks = (N + BK - 1) / BK;
  ga.kb_per_split = (ga.kblocks + nsplit - 1) / nsplit;
  ga.nsplit = nsplit;
  ga.gpart = gpart;
  ga.limit_ns = la.limit_ns;
  gram_tc_kernel<<<dim3((C + G_ROWS - 1) / G_ROWS, nsplit), THREADS, gsmem, stream>>>(mHi, mLo, ga);
  OM_LAUNCHED("gram_tc_kernel");
  return ORDERMOE_OK;
}

}  // namespace om
