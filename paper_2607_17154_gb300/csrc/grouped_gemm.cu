// Grouped SwiGLU expert FFN on sm_103a tensor cores (tcgen05 + TMEM + TMA).
//
// Persistent warp-specialised kernels over the expert-contiguous rows of
// ordermoe_dispatch, with the per-expert row ranges read on the device: a
// one-CTA kernel for small batches (described here) and a CTA-pair kernel
// with the weights on the MMA's M side for large ones (its own section below).
// One-CTA kernel:
//   gate/up: H[rows of e, n0:n0+128] = bf16(silu(X W1_e^T) * (X W3_e^T)) for a
//            128-column slice n0 of d_ff. One tcgen05.mma of N = 256 computes
//            the gate (TMEM columns 0..127) and up (128..255) projections from
//            a B tile whose first 128 rows are W1_e rows and last 128 rows are
//            W3_e rows; the epilogue fuses SwiGLU.
//   down:    Y[rows of e, n0:n0+256] = bf16(H W2_e^T).
// Tile = 128 rows x 256 accumulator columns, K step 64 (one 128-byte
// swizzled TMA box per operand row), 4-stage shared-memory ring, two TMEM
// accumulators (2 x 256 columns = all 512) so the epilogue of one tile
// overlaps the main loop of the next.
// Warp roles (192 threads): warp 0 = TMA producer, warp 1 = MMA issuer and
// TMEM owner, warps 2-5 = epilogue (warp w reads TMEM lanes 32 (w % 4) ...).
// Tile order: expert, then N slice, then M tile, so CTAs running at the same
// time share the same weight slice through L2.
// Every wait is bounded (globaltimer); a wait that runs out reports
// ORDERMOE_DEV_WAIT_TIMEOUT, makes the other roles stop, drains the copies
// and MMAs in flight (bounded too), frees TMEM and returns.
#include <initializer_list>
#include <mutex>

#include "common.cuh"

namespace om {

static __device__ unsigned long long g_err_gemm = 0;

int read_clear_err_gemm(unsigned long long* out) {
  unsigned long long zero = 0;
  OM_CUDA(cudaMemcpyFromSymbol(out, g_err_gemm, sizeof(*out)));
  OM_CUDA(cudaMemcpyToSymbol(g_err_gemm, &zero, sizeof(zero)));
  return ORDERMOE_OK;
}

namespace gg {

constexpr int BM = 128;
constexpr int BN = 256;  // accumulator columns per tile
constexpr int BK = 64;   // bf16 elements = 128 bytes
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int BOX_BYTES = 128 * BK * 2;  // one TMA box: 128 rows x 64 columns
constexpr int THREADS = 192;
constexpr int TMEM_COLS = 512;
constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN);

struct Smem {
  uint64_t full[STAGES];
  uint64_t empty[STAGES];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
  int zero;
  int mt_start[ORDERMOE_MAX_EXPERTS + 1];
  int offs[ORDERMOE_MAX_EXPERTS + 1];
};
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + static_cast<int>(sizeof(Smem));

enum { GATEUP = 0, DOWN = 1, LOGITS = 2 };

struct Args {
  const int32_t* offsets;  // [E+1] row ranges (0 <= ... <= rows); null: one group of `rows` rows
  int rows;
  int n_valid;       // LOGITS: number of valid output columns
  float* out_f32;    // LOGITS: H [rows][n_valid] fp32
  int E;
  int K;             // reduction length
  int n_tiles;       // N slices per expert
  int b_rows;        // weight rows per expert in the B tensor map (d_ff or d)
  uint16_t* out;     // H [R][d_ff] or Y [R][d]
  int ldo;           // row length of out
  uint64_t limit_ns; // bounded-wait limit
  int m_major;       // 1: all N slices of an M tile back to back (A read once from HBM)
};

struct Tile {
  int e, m0, m_end, n;
};

__device__ __forceinline__ Tile decode(int tile, const Smem& s, int E, int n_tiles, int m_major) {
  // the last expert whose first tile is <= tile (binary search: the row-tile
  // starts never decrease; empty experts share their successor's start)
  int e = 0, hi = E - 1;
  while (e < hi) {
    const int mid = (e + hi + 1) >> 1;
    if (s.mt_start[mid] * n_tiles <= tile) e = mid;
    else hi = mid - 1;
  }
  const int local = tile - s.mt_start[e] * n_tiles;
  const int n_mt = s.mt_start[e + 1] - s.mt_start[e];
  Tile t;
  t.e = e;
  int mt;
  if (m_major) {
    mt = local / n_tiles;
    t.n = local - mt * n_tiles;
  } else {
    t.n = local / n_mt;
    mt = local - t.n * n_mt;
  }
  t.m0 = s.offs[e] + mt * BM;
  t.m_end = s.offs[e + 1];
  return t;
}

template <int MODE>
__global__ void __launch_bounds__(THREADS, 1)
    ffn_gemm_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB0,
                    const __grid_constant__ CUtensorMap mapB1, Args args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* tiles = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  Smem& s = *reinterpret_cast<Smem*>(tiles + STAGES * STAGE_BYTES);
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  // launched with launch_pdl: barriers, TMEM and tensor-map prefetches are set
  // up while the previous kernel finishes; global memory only after pdl_wait
  pdl_trigger();
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&mapA);
    tma_prefetch_map(&mapB0);
    if (MODE == GATEUP) tma_prefetch_map(&mapB1);
  }

  if (tid == 0) {
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.tfull[i], 1);
      mbar_init(&s.tempty[i], 128);
    }
    mbar_init(&s.drain, 1);
    s.abort = 0;
    s.zero = 0;
    pdl_wait();  // the offsets come from the permutation
    int acc = 0;
    bool bad = false;
    for (int e = 0; e <= args.E; ++e) {
      const int o = args.offsets ? args.offsets[e] : (e == 0 ? 0 : args.rows);
      s.offs[e] = o;
      if (e == 0 && o != 0) bad = true;
      if (e > 0) {
        const int rows = o - s.offs[e - 1];
        if (rows < 0) bad = true;
        acc += rows > 0 ? (rows + BM - 1) / BM : 0;
      }
      s.mt_start[e] = acc;
    }
    if (bad || s.offs[args.E] > args.rows) {  // offsets must run 0 <= ... <= rows
      if (blockIdx.x == 0) report(&g_err_gemm, ORDERMOE_DEV_BAD_INDEX, -2);
      for (int e = 0; e <= args.E; ++e) s.mt_start[e] = 0;  // no tiles
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&s.tmem_base, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();  // every thread: the previous kernel's outputs are visible
  const uint32_t tmem_base = s.tmem_base;
  const int total = s.mt_start[args.E] * args.n_tiles;
  const int kblocks = args.K / BK;
  volatile int* abort = &s.abort;

  // per-role bookkeeping for the drain after an abort
  uint32_t issued_mask = 0, last_phase_bits = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (int tile = blockIdx.x; tile < total && !*abort; tile += gridDim.x) {
        const Tile t = decode(tile, s, args.E, args.n_tiles, args.m_major);
        const int brow = t.e * args.b_rows + t.n * (MODE == GATEUP ? 128 : 256);  // LOGITS: e == 0
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&s.empty[stage], phase ^ 1u, args.limit_ns, abort)) {
            if (!*abort) report(&g_err_gemm, ORDERMOE_DEV_WAIT_TIMEOUT, 1);
            *abort = 1;
            break;
          }
          uint8_t* sa = tiles + stage * STAGE_BYTES;
          uint8_t* sb = sa + A_BYTES;
          mbar_arrive_expect_tx(&s.full[stage], STAGE_BYTES);
          tma_load_2d(sa, &mapA, &s.full[stage], kb * BK, t.m0);
          if (MODE == GATEUP) {
            tma_load_2d(sb, &mapB0, &s.full[stage], kb * BK, brow);
            tma_load_2d(sb + BOX_BYTES, &mapB1, &s.full[stage], kb * BK, brow);
          } else {
            tma_load_2d(sb, &mapB0, &s.full[stage], kb * BK, brow);
            tma_load_2d(sb + BOX_BYTES, &mapB0, &s.full[stage], kb * BK, brow + 128);
          }
          issued_mask |= 1u << stage;
          last_phase_bits = (last_phase_bits & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int tile = blockIdx.x; tile < total && !*abort; tile += gridDim.x, ++it) {
        const int slot = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait(&s.tempty[slot], acc_phase ^ 1u, args.limit_ns, abort)) {
          if (!*abort) report(&g_err_gemm, ORDERMOE_DEV_WAIT_TIMEOUT, 2);
          *abort = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + slot * BN;
        bool ok = true;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&s.full[stage], phase, args.limit_ns, abort)) {
            if (!*abort) report(&g_err_gemm, ORDERMOE_DEV_WAIT_TIMEOUT, 3);
            *abort = 1;
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(tiles + stage * STAGE_BYTES);
          const uint32_t b0 = a0 + A_BYTES;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            mma_bf16(d_tmem, sdesc_kmajor_sw128(a0 + kk * 32), sdesc_kmajor_sw128(b0 + kk * 32),
                     IDESC, (kb | kk) != 0 ? 1u : 0u);
          }
          mma_issued = true;
          mma_commit(&s.empty[stage]);
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        mma_commit(&s.tfull[slot]);
      }
    }
  } else {
    // epilogue: warps 2..5 -> TMEM lane quarter (warp % 4)
    const int q = warp & 3;
    const int lrow = q * 32 + lane;
    int it = 0;
    for (int tile = blockIdx.x; tile < total; tile += gridDim.x, ++it) {
      // warp-uniform control flow: tcgen05.ld below is .sync.aligned
      if (__any_sync(0xffffffffu, *abort != 0)) break;
      const int slot = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&s.tfull[slot], acc_phase, args.limit_ns, abort));
      if (!ok) {
        if (lane == 0 && !*abort) report(&g_err_gemm, ORDERMOE_DEV_WAIT_TIMEOUT, 4);
        *abort = 1;
        break;
      }
      tc_fence_after();
      const Tile t = decode(tile, s, args.E, args.n_tiles, args.m_major);
      const int row = t.m0 + lrow;
      const bool valid = row < t.m_end;
      const uint32_t tb = tmem_base + slot * BN + (static_cast<uint32_t>(q * 32) << 16);
      if (MODE == GATEUP) {
        uint16_t* orow = args.out + (size_t)row * args.ldo + t.n * 128;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t g[32], u[32];
          tmem_ld32(tb + c * 32, g);
          tmem_ld32(tb + 128 + c * 32, u);
          tmem_ld_wait();
          if (valid) {
            uint32_t pk[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const float g0 = __uint_as_float(g[2 * i]), g1 = __uint_as_float(g[2 * i + 1]);
              const float u0 = __uint_as_float(u[2 * i]), u1 = __uint_as_float(u[2 * i + 1]);
              const float h0 = g0 / (1.0f + __expf(-g0)) * u0;
              const float h1 = g1 / (1.0f + __expf(-g1)) * u1;
              pk[i] = pack_bf16x2(h0, h1);
            }
            uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
            for (int i = 0; i < 4; ++i)
              dst[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
          }
        }
      } else if (MODE == LOGITS) {
        const int col0 = t.n * 256;
        float* orow = args.out_f32 + (size_t)row * args.n_valid;
        const bool vec = (args.n_valid & 3) == 0;
#pragma unroll 1
        for (int c = 0; c < 8; ++c) {
          if (col0 + c * 32 >= args.n_valid) break;  // warp-uniform
          uint32_t v[32];
          tmem_ld32(tb + c * 32, v);
          tmem_ld_wait();
          if (valid) {
            const int cb = col0 + c * 32;
            if (vec && cb + 32 <= args.n_valid) {
              float4* dst = reinterpret_cast<float4*>(orow + cb);
#pragma unroll
              for (int i = 0; i < 8; ++i)
                dst[i] = make_float4(__uint_as_float(v[4 * i]), __uint_as_float(v[4 * i + 1]),
                                     __uint_as_float(v[4 * i + 2]), __uint_as_float(v[4 * i + 3]));
            } else {
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (cb + i < args.n_valid) orow[cb + i] = __uint_as_float(v[i]);
            }
          }
        }
      } else {
        uint16_t* orow = args.out + (size_t)row * args.ldo + t.n * 256;
#pragma unroll 1
        for (int c = 0; c < 8; ++c) {
          uint32_t v[32];
          tmem_ld32(tb + c * 32, v);
          tmem_ld_wait();
          if (valid) {
            uint32_t pk[16];
#pragma unroll
            for (int i = 0; i < 16; ++i)
              pk[i] = pack_bf16x2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
            uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
            for (int i = 0; i < 4; ++i)
              dst[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
          }
        }
      }
      tc_fence_before();
      mbar_arrive(&s.tempty[slot]);
    }
  }

  __syncthreads();
  if (s.abort) {
    volatile int* never = &s.zero;
    if (warp == 0 && lane == 0) {
      // wait for every TMA copy this CTA issued (bounded)
      for (int st = 0; st < STAGES; ++st)
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
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ------------------------------------------------- CTA-pair variant (gate/up, down)
//
// A pair of CTAs on 2 SMs computes, with tcgen05.mma.cta_group::2 issued
// by the even CTA, a tile of 256 weight rows (the MMA's M side; 128 in each
// CTA's shared memory and TMEM lanes) by up to 256 permuted rows of one expert
// (the N side, split evenly between the two CTAs' shared memory). The weight
// side is always full; an expert's last row tile is cut to the next multiple of
// 16 rows (the N granularity of the instruction), so at most 15 padding rows
// are computed per expert instead of up to 255 for a 256-row M tile. Each CTA
// loads its rows as one 128-row TMA box (of which the MMA reads the first N/2):
// a stage of 5-6 smaller boxes starved the tensor pipe.
//   gate/up: CTA r holds W1_e rows f..f+63 (TMEM lanes 0..63) and the same
//            rows of W3_e (lanes 64..127), f = 128 n + 64 r; the epilogue
//            warps of the gate and up lanes exchange half of their values
//            through shared memory and each forms SwiGLU for half the rows.
//   down:    CTA r holds W2_e rows 256 n + 128 r + 0..127 (all 128 lanes).
// The accumulator is transposed (lane = output column, TMEM column = row);
// the epilogue writes it row-major through a shared-memory tile with 16-byte
// coalesced stores, skipping rows beyond the expert's range.
// Each cluster is one CTA pair, and each CTA loads its own operand boxes from
// this GPU's memory (no multicast loads).
// Barriers: full[s] (even CTA, one arrive with the pair's bytes; both CTAs'
// TMA loads complete on it), empty[s] and tfull[b] (both CTAs, arrived by the
// even CTA's MMA commits signalled to the pair), tempty[b] (even CTA, one
// arrive per epilogue warp of either CTA). The gate/up epilogue runs on two
// groups of four warps that take alternate 32-row chunks, so two chunks are
// in flight (short-K tiles are otherwise epilogue-bound); down runs one group.
// Named barriers 1 and 2 (the 128 threads of a group) order each group's
// shared-memory exchange, and the decision to stop is a barrier reduction over
// all epilogue warps (barrier 3), so they always leave together.
constexpr int P_BM = 256;            // permuted rows (N side) per tile
constexpr int P_MAX_STAGES = 6;
constexpr int P_W_BYTES = 128 * BK * 2;   // 128 weight rows per CTA and K block
constexpr int P_T_BYTES = 128 * BK * 2;   // one box of 128 permuted rows per CTA
constexpr int P_STAGE_BYTES = P_W_BYTES + P_T_BYTES;
constexpr int P_X_PITCH = 17;             // floats per exchange row (odd: no bank conflicts)
constexpr int P_XBUF_FLOATS = 128 * P_X_PITCH;
constexpr int P_EPI_GROUP_BYTES = 2 * (P_XBUF_FLOATS * 4 + 32 * 64 * 2);  // gate/up, double-buffered
static_assert(P_EPI_GROUP_BYTES >= 2 * 32 * 128 * 2, "down staging fits");


struct PSmem {
  uint64_t full[P_MAX_STAGES];
  uint64_t empty[P_MAX_STAGES];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
  int zero;
  int mt_start[ORDERMOE_MAX_EXPERTS + 1];
  int offs[ORDERMOE_MAX_EXPERTS + 1];
};
// Per projection: gate/up (SwiGLU exchange in the epilogue) runs two epilogue
// groups of four warps and five stages; down (a plain conversion) one group
// and six stages. Five stages time the same as six for gate/up, and a second
// group made down slower.
template <int MODE>
struct PCfg {
  static constexpr int GROUPS = MODE == GATEUP ? 2 : 1;
  static constexpr int EPI_WARPS = 4 * GROUPS;
  static constexpr int THREADS = 64 + 32 * EPI_WARPS;
  static constexpr int STAGES = MODE == GATEUP ? 5 : 6;
  static constexpr int EPI_BYTES = GROUPS * P_EPI_GROUP_BYTES;
  static constexpr int SMEM_BYTES =
      STAGES * P_STAGE_BYTES + EPI_BYTES + 1024 + static_cast<int>(sizeof(PSmem));
  static_assert(STAGES <= P_MAX_STAGES, "stage barriers");
  static_assert(SMEM_BYTES <= 227 * 1024, "pair kernel shared memory");
};

__device__ __forceinline__ Tile decode_pair(int tile, const PSmem& s, int E, int n_tiles) {
  // the last expert whose first tile is <= tile (binary search: the row-tile
  // starts never decrease; empty experts share their successor's start)
  int e = 0, hi = E - 1;
  while (e < hi) {
    const int mid = (e + hi + 1) >> 1;
    if (s.mt_start[mid] * n_tiles <= tile) e = mid;
    else hi = mid - 1;
  }
  const int local = tile - s.mt_start[e] * n_tiles;
  const int n_mt = s.mt_start[e + 1] - s.mt_start[e];
  Tile t;
  t.e = e;
  t.n = local / n_mt;
  t.m0 = s.offs[e] + (local - t.n * n_mt) * P_BM;
  t.m_end = s.offs[e + 1];
  return t;
}

// rows of the tile rounded up to the MMA's N granularity (16)
__device__ __forceinline__ int tile_n(const Tile& t) {
  const int rows = min(P_BM, t.m_end - t.m0);
  return (rows + 15) & ~15;
}

// the 128 threads of epilogue group grp (named barriers 1 and 2)
__device__ __forceinline__ void epi_sync(int grp) {
  asm volatile("bar.sync %0, 128;" ::"r"(1 + grp) : "memory");
}
// true in every epilogue thread iff p holds in all N of them (named barrier 3)
template <int N>
__device__ __forceinline__ bool epi_all(bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.and.pred po, 3, %2, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(p)), "n"(N)
      : "memory");
  return r != 0;
}

// Tensor maps of the permuted rows with boxes of 16, 32, ..., 128 rows: a
// tile cut to N rows loads N/2 rows per CTA (rounded up to 16) instead of a
// full 128-row box, since it is the row boxes, not the MMAs, that bound a
// cut tile (an expert's last one).
struct RowMaps {
  CUtensorMap m[8];  // m[i]: box of 16 (i + 1) rows
};

// One cluster = one CTA pair.
template <int MODE>
__global__ void __launch_bounds__(PCfg<MODE>::THREADS, 1)
    ffn_gemm_pair_kernel(const __grid_constant__ CUtensorMap mapW0,
                         const __grid_constant__ CUtensorMap mapW1,
                         const __grid_constant__ RowMaps mapT, Args args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* tiles = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  constexpr int P_STAGES = PCfg<MODE>::STAGES;
  uint8_t* epi = tiles + P_STAGES * P_STAGE_BYTES;
  PSmem& s = *reinterpret_cast<PSmem*>(epi + PCfg<MODE>::EPI_BYTES);
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const uint32_t rank = cluster_ctarank();
  const uint32_t rp = rank & 1u;     // rank within the pair
  const uint32_t lead = 0;           // the pair's even CTA (MMA issuer)
  const bool even = (rp == 0);
  const int cluster = blockIdx.x / 2;
  const int n_clusters = gridDim.x / 2;
  // launched with launch_pdl: barriers, TMEM and tensor-map prefetches are set
  // up while the previous kernel finishes; global memory only after pdl_wait
  pdl_trigger();
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&mapW0);
    if (MODE == GATEUP) tma_prefetch_map(&mapW1);
#pragma unroll
    for (int i = 0; i < 8; ++i) tma_prefetch_map(&mapT.m[i]);
  }

  if (tid == 0) {
    for (int i = 0; i < P_STAGES; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 1);  // one MMA commit of the pair
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.tfull[i], 1);
      mbar_init(&s.tempty[i], 2 * PCfg<MODE>::EPI_WARPS);  // every epilogue warp of both CTAs
    }
    mbar_init(&s.drain, 1);
    s.abort = 0;
    s.zero = 0;
    pdl_wait();  // the offsets come from the permutation
    int acc = 0;
    bool bad = false;
    for (int e = 0; e <= args.E; ++e) {
      const int o = args.offsets[e];
      s.offs[e] = o;
      if (e == 0 && o != 0) bad = true;
      if (e > 0) {
        const int rows = o - s.offs[e - 1];
        if (rows < 0) bad = true;
        acc += rows > 0 ? (rows + P_BM - 1) / P_BM : 0;
      }
      s.mt_start[e] = acc;
    }
    if (bad || s.offs[args.E] > args.rows) {
      if (blockIdx.x == 0) report(&g_err_gemm, ORDERMOE_DEV_BAD_INDEX, -2);
      for (int e = 0; e <= args.E; ++e) s.mt_start[e] = 0;
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(&s.tmem_base, TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();  // barriers of both CTAs initialised, TMEM allocated
  tc_fence_after();
  pdl_wait();  // every thread: the previous kernel's outputs are visible
  const uint32_t tmem_base = s.tmem_base;
  const int total = s.mt_start[args.E] * args.n_tiles;
  const int kblocks = args.K / BK;
  volatile int* abort = &s.abort;
  uint32_t issued_mask = 0, last_phase_bits = 0;
  bool mma_issued = false;
  // tile -> (expert, column slice, row range)
  auto tile_of = [&](int tile) { return decode_pair(tile, s, args.E, args.n_tiles); };

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (int tile = cluster; tile < total && !*abort; tile += n_clusters) {
        const Tile t = tile_of(tile);
        const int trow = t.m0 + static_cast<int>(rp) * (tile_n(t) >> 1);  // N/2 rows per CTA
        const int hb = ((tile_n(t) >> 1) + 15) & ~15;  // rows per CTA's box (16 .. 128)
        const CUtensorMap* mrow = &mapT.m[(hb >> 4) - 1];
        const uint32_t stage_tx = 2u * static_cast<uint32_t>(P_W_BYTES + hb * BK * 2);
        const int wrow = (MODE == GATEUP)
                             ? t.e * args.b_rows + t.n * 128 + 64 * static_cast<int>(rp)
                             : t.e * args.b_rows + t.n * 256 + 128 * static_cast<int>(rp);
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&s.empty[stage], phase ^ 1u, args.limit_ns, abort)) {
            if (!*abort) report(&g_err_gemm, ORDERMOE_DEV_WAIT_TIMEOUT, 11);
            *abort = 1;
            break;
          }
          uint8_t* sw = tiles + stage * P_STAGE_BYTES;
          uint8_t* st = sw + P_W_BYTES;
          const uint32_t full_even = mapa_shared(smem_u32(&s.full[stage]), lead);
          if (even) mbar_arrive_expect_tx(&s.full[stage], stage_tx);
          if (MODE == GATEUP) {
            tma_load_2d_pair(sw, &mapW0, full_even, kb * BK, wrow);             // W1: lanes 0..63
            tma_load_2d_pair(sw + P_W_BYTES / 2, &mapW1, full_even, kb * BK, wrow);  // W3: 64..127
          } else {
            tma_load_2d_pair(sw, &mapW0, full_even, kb * BK, wrow);
          }
          tma_load_2d_pair(st, mrow, full_even, kb * BK, trow);
          issued_mask |= 1u << stage;
          last_phase_bits = (last_phase_bits & ~(1u << stage)) | (phase << stage);
          if (++stage == P_STAGES) { stage = 0; phase ^= 1u; }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && even) {
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int tile = cluster; tile < total && !*abort; tile += n_clusters, ++it) {
        const int slot = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait(&s.tempty[slot], acc_phase ^ 1u, args.limit_ns, abort)) {
          if (!*abort) report(&g_err_gemm, ORDERMOE_DEV_WAIT_TIMEOUT, 12);
          *abort = 1;
          break;
        }
        tc_fence_after();
        const Tile t = tile_of(tile);
        const uint32_t idesc = idesc_bf16_f32(256, tile_n(t));
        const uint32_t d_tmem = tmem_base + slot * BN;
        bool ok = true;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&s.full[stage], phase, args.limit_ns, abort)) {
            if (!*abort) report(&g_err_gemm, ORDERMOE_DEV_WAIT_TIMEOUT, 13);
            *abort = 1;
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(tiles + stage * P_STAGE_BYTES);
          const uint32_t b0 = a0 + P_W_BYTES;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            mma_bf16_pair(d_tmem, sdesc_kmajor_sw128(a0 + kk * 32),
                          sdesc_kmajor_sw128(b0 + kk * 32), idesc, (kb | kk) != 0 ? 1u : 0u);
          mma_issued = true;
          mma_commit_pair(&s.empty[stage], 0x3);
          if (++stage == P_STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        mma_commit_pair(&s.tfull[slot], 0x3);
      }
    }
  } else {
    // epilogue: warps 2..9 in two groups of four; TMEM lane quarter q = warp % 4;
    // group grp takes the 32-row chunks grp, grp + 2, ... of every tile
    const int q = warp & 3;
    const int grp = (warp - 2) >> 2;  // 0 .. GROUPS - 1
    const int et = tid - 64 - 128 * grp;  // 0..127 within the group
    uint8_t* ge = epi + grp * P_EPI_GROUP_BYTES;
    float* xbuf = reinterpret_cast<float*>(ge);                          // [2][128][P_X_PITCH]
    uint16_t* obuf = reinterpret_cast<uint16_t*>(ge + 2 * P_XBUF_FLOATS * 4);  // gate/up [2][32][64]
    uint16_t* ybuf = reinterpret_cast<uint16_t*>(ge);                    // down [2][32][128]
    int it = 0;
    for (int tile = cluster; tile < total; tile += n_clusters, ++it) {
      const int slot = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const bool waited = (*abort == 0) && mbar_wait(&s.tfull[slot], acc_phase, args.limit_ns, abort);
      if (!epi_all<PCfg<MODE>::EPI_WARPS * 32>(waited)) {  // the same decision in every epilogue warp
        if (!waited && lane == 0 && !*abort) report(&g_err_gemm, ORDERMOE_DEV_WAIT_TIMEOUT, 14);
        *abort = 1;
        break;
      }
      tc_fence_after();
      const Tile t = tile_of(tile);
      const int rows = min(P_BM, t.m_end - t.m0);
      const int nchunks = (rows + 31) >> 5;
      const uint32_t tb = tmem_base + slot * BN + (static_cast<uint32_t>(q * 32) << 16);
#pragma unroll 1
      for (int c = grp; c < nchunks; c += PCfg<MODE>::GROUPS) {
        const int buf = (c / PCfg<MODE>::GROUPS) & 1;
        uint32_t v[32];
        tmem_ld32(tb + c * 32, v);  // TMEM column = row c*32 + i of the tile
        tmem_ld_wait();
        if (MODE == GATEUP) {
          // gate lanes (q 0, 1) keep rows 0..15 of the chunk and hand 16..31
          // to the up lanes (q 2, 3) of the same columns, which hand back 0..15
          const bool gate = q < 2;
          const int keep = gate ? 0 : 16;
          float* xb = xbuf + buf * P_XBUF_FLOATS;
          float* mine = xb + (q * 32 + lane) * P_X_PITCH;
#pragma unroll
          for (int i = 0; i < 16; ++i) mine[i] = __uint_as_float(gate ? v[16 + i] : v[i]);
          epi_sync(grp);
          const float* other = xb + ((q ^ 2) * 32 + lane) * P_X_PITCH;
          uint16_t* ob = obuf + buf * (32 * 64);
          const int col = (q & 1) * 32 + lane;
#pragma unroll
          for (int i = 0; i < 16; i += 2) {
            float h[2];
#pragma unroll
            for (int j = 0; j < 2; ++j) {
              const float own = __uint_as_float(gate ? v[i + j] : v[16 + i + j]);
              const float oth = other[i + j];
              const float g = gate ? own : oth;
              const float u = gate ? oth : own;
              // silu(g) u = g u / (1 + e^-g); the quotient by the fast reciprocal
              // (2 ulp in fp32, far below the bf16 rounding of h)
              h[j] = __fdividef(g * u, 1.0f + __expf(-g));
            }
            const uint32_t pk = pack_bf16x2(h[0], h[1]);
            ob[(keep + i) * 64 + col] = static_cast<uint16_t>(pk & 0xFFFFu);
            ob[(keep + i + 1) * 64 + col] = static_cast<uint16_t>(pk >> 16);
          }
          epi_sync(grp);
          uint16_t* gcol = args.out + t.n * 128 + 64 * static_cast<int>(rp) + (et & 7) * 8;
#pragma unroll
          for (int p = 0; p < 2; ++p) {
            const int r = p * 16 + (et >> 3);
            const int row = c * 32 + r;
            if (row < rows)
              *reinterpret_cast<uint4*>(gcol + (size_t)(t.m0 + row) * args.ldo) =
                  *reinterpret_cast<const uint4*>(ob + r * 64 + (et & 7) * 8);
          }
        } else {
          uint16_t* yb = ybuf + buf * (32 * 128);
          const int col = q * 32 + lane;
#pragma unroll
          for (int i = 0; i < 32; i += 2) {
            const uint32_t pk = pack_bf16x2(__uint_as_float(v[i]), __uint_as_float(v[i + 1]));
            yb[i * 128 + col] = static_cast<uint16_t>(pk & 0xFFFFu);
            yb[(i + 1) * 128 + col] = static_cast<uint16_t>(pk >> 16);
          }
          epi_sync(grp);
          uint16_t* gcol = args.out + t.n * 256 + 128 * static_cast<int>(rp) + (et & 15) * 8;
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const int r = p * 8 + (et >> 4);
            const int row = c * 32 + r;
            if (row < rows)
              *reinterpret_cast<uint4*>(gcol + (size_t)(t.m0 + row) * args.ldo) =
                  *reinterpret_cast<const uint4*>(yb + r * 128 + (et & 15) * 8);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(mapa_shared(smem_u32(&s.tempty[slot]), lead));
    }
  }

  __syncthreads();
  if (s.abort) {
    volatile int* never = &s.zero;
    if (warp == 0 && lane == 0 && even) {
      for (int st = 0; st < P_STAGES; ++st)
        if ((issued_mask >> st) & 1u)
          mbar_wait(&s.full[st], (last_phase_bits >> st) & 1u, args.limit_ns, never);
    }
    if (warp == 1 && lane == 0 && even && mma_issued) {
      mma_commit_pair(&s.drain, static_cast<uint16_t>(1u << rank));
      mbar_wait(&s.drain, 0, args.limit_ns, never);
    }
  }
  tc_fence_before();
  cluster_sync();  // every CTA finished: no more arrivals or copies into any
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem_base, TMEM_COLS);
}

// ------------------------------------------------------------------- host
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// 2-D bf16 row-major [rows][cols] map with a 64 x 128 box and 128-byte swizzle.
int make_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols) {
  return make_tmap_bf16(map, base, rows, cols, 128);
}

}  // namespace gg

int make_tmap_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols,
                   uint32_t box_rows) {
  gg::EncodeTiledFn enc = gg::encode_fn();
  if (!enc) return fail(ORDERMOE_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {gg::BK, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(ORDERMOE_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return ORDERMOE_OK;
}

template <int MODE>
static cudaError_t pair_attr() {
  return cudaFuncSetAttribute(gg::ffn_gemm_pair_kernel<MODE>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                              gg::PCfg<MODE>::SMEM_BYTES);
}

static int ffn_attrs() {
  using namespace gg;
  static PerDevice cache;
  const cudaError_t attr_err = static_cast<cudaError_t>(per_device(cache, [] {
    cudaError_t e = pair_attr<GATEUP>();
    if (e == cudaSuccess) e = pair_attr<DOWN>();
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(ffn_gemm_kernel<GATEUP>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(ffn_gemm_kernel<DOWN>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    return static_cast<int>(e);
  }));
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(ffn_gemm_pair_kernel)");
  return ORDERMOE_OK;
}

template <int MODE>
static cudaLaunchConfig_t pair_config(int grid, int cl, cudaStream_t stream,
                                      cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(gg::PCfg<MODE>::THREADS, 1, 1);
  cfg.dynamicSmemBytes = gg::PCfg<MODE>::SMEM_BYTES;
  cfg.stream = stream;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cl;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // waits in the kernel
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_on(stream) ? 2 : 1;
  return cfg;
}

// CTA pairs that can be resident at once (not every SM finds a partner in its
// GPC: 76 pairs on GB300); the persistent grid never exceeds it, so no
// cluster waits for another.
template <int MODE>
static int max_resident_clusters() {
  static PerDevice cache;
  return per_device(cache, [] {
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = pair_config<MODE>(2 * (num_sms() / 2), 2, nullptr, attr);
    cfg.numAttrs = 1;  // the cluster shape alone decides residency
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gg::ffn_gemm_pair_kernel<MODE>, &cfg) != cudaSuccess ||
        n <= 0) {
      cudaGetLastError();
      n = num_sms() / 2;
    }
    return n < num_sms() / 2 ? n : num_sms() / 2;
  });
}

// One launch of the CTA-pair kernel over `tiles` pair tiles.
template <int MODE>
static int launch_pair(const CUtensorMap& w0, const CUtensorMap& w1, const gg::RowMaps& t,
                       const gg::Args& a, long long tiles, cudaStream_t stream, const char* what) {
  const long long cmax = max_resident_clusters<MODE>();
  const long long clusters = tiles < cmax ? tiles : cmax;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg =
      pair_config<MODE>(static_cast<int>(2 * (clusters > 0 ? clusters : 1)), 2, stream, attr);
  const cudaError_t e = cudaLaunchKernelEx(&cfg, gg::ffn_gemm_pair_kernel<MODE>, w0, w1, t, a);
  if (e != cudaSuccess) return cuda_fail(e, what);
  OM_LAUNCHED(what);
  return ORDERMOE_OK;
}

// The row maps of a [rows][cols] bf16 tensor, boxes of 16 .. 128 rows.
static int make_row_maps(gg::RowMaps* rm, const void* base, uint64_t rows, uint64_t cols) {
  for (int i = 0; i < 8; ++i) {
    const int rc = make_tmap_bf16(&rm->m[i], base, rows, cols, static_cast<uint32_t>(16 * (i + 1)));
    if (rc) return rc;
  }
  return ORDERMOE_OK;
}

// Tile shape: CTA pairs (256 weight rows x up to 256 permuted rows) when experts average at least 256 rows; otherwise single
// CTAs with 128-row tiles and the rows on the M side (a decode step: ~32 rows
// per expert, where the weights are streamed once and the MMA shape hardly
// matters).
static bool use_pairs(int R, int E) { return (long long)R >= 256LL * E; }

static int single_grid(long long tiles) {
  const int sms = num_sms();
  return static_cast<int>(tiles < sms ? tiles : sms);
}

// H = SwiGLU(X_perm W1^T, X_perm W3^T) over the expert row ranges.
int gate_up_launch(const uint16_t* X_perm, const int32_t* offsets, int R, const uint16_t* W1,
                   const uint16_t* W3, int E, int d, int dff, uint16_t* H, cudaStream_t stream) {
  using namespace gg;
  int rc;
  if ((rc = ffn_attrs())) return rc;
  Args a{};
  a.offsets = offsets; a.rows = R; a.E = E; a.limit_ns = wait_limit_ns();
  a.K = d; a.n_tiles = dff / 128; a.b_rows = dff; a.out = H; a.ldo = dff;
  CUtensorMap mX, mW1, mW3;
  if ((rc = make_map(&mX, X_perm, R, d))) return rc;
  if (use_pairs(R, E)) {
    // weights on the MMA's M side in 64-row boxes of W1 and W3
    if ((rc = make_tmap_bf16(&mW1, W1, (uint64_t)E * dff, d, 64))) return rc;
    if ((rc = make_tmap_bf16(&mW3, W3, (uint64_t)E * dff, d, 64))) return rc;
    const long long row_tiles = (long long)(R + P_BM - 1) / P_BM + E;
    gg::RowMaps rX;
    if ((rc = make_row_maps(&rX, X_perm, R, d))) return rc;
    return launch_pair<GATEUP>(mW1, mW3, rX, a, row_tiles * a.n_tiles, stream,
                               "ffn_gemm_pair_kernel<gate_up>");
  } else {
    if ((rc = make_map(&mW1, W1, (uint64_t)E * dff, d))) return rc;
    if ((rc = make_map(&mW3, W3, (uint64_t)E * dff, d))) return rc;
    const long long tiles = ((long long)(R + BM - 1) / BM + E) * a.n_tiles;
    OM_LAUNCH_PDL("ffn_gemm_kernel<gate_up>", ffn_gemm_kernel<GATEUP>, dim3(single_grid(tiles)),
                  dim3(THREADS), SMEM_BYTES, stream, mX, mW1, mW3, a);
  }
  return ORDERMOE_OK;
}

// Y_perm = H W2^T over the expert row ranges.
int down_launch(const uint16_t* H, const int32_t* offsets, int R, const uint16_t* W2, int E, int d,
                int dff, uint16_t* Y, cudaStream_t stream) {
  using namespace gg;
  int rc;
  if ((rc = ffn_attrs())) return rc;
  Args a{};
  a.offsets = offsets; a.rows = R; a.E = E; a.limit_ns = wait_limit_ns();
  a.K = dff; a.n_tiles = d / 256; a.b_rows = d; a.out = Y; a.ldo = d;
  CUtensorMap mH, mW2;
  if ((rc = make_map(&mW2, W2, (uint64_t)E * d, dff))) return rc;
  if ((rc = make_map(&mH, H, R, dff))) return rc;
  if (use_pairs(R, E)) {
    const long long row_tiles = (long long)(R + P_BM - 1) / P_BM + E;
    gg::RowMaps rH;
    if ((rc = make_row_maps(&rH, H, R, dff))) return rc;
    return launch_pair<DOWN>(mW2, mW2, rH, a, row_tiles * a.n_tiles, stream,
                             "ffn_gemm_pair_kernel<down>");
  } else {
    const long long tiles = ((long long)(R + BM - 1) / BM + E) * a.n_tiles;
    OM_LAUNCH_PDL("ffn_gemm_kernel<down>", ffn_gemm_kernel<DOWN>, dim3(single_grid(tiles)),
                  dim3(THREADS), SMEM_BYTES, stream, mH, mW2, mW2, a);
  }
  return ORDERMOE_OK;
}

int ffn_launch(const uint16_t* X_perm, const int32_t* offsets, int R, const uint16_t* W1,
               const uint16_t* W3, const uint16_t* W2, int E, int d, int dff, uint16_t* H,
               uint16_t* Y, cudaStream_t stream) {
  int rc = gate_up_launch(X_perm, offsets, R, W1, W3, E, d, dff, H, stream);
  if (rc) return rc;
  return down_launch(H, offsets, R, W2, E, d, dff, Y, stream);
}

// H[n][c] = sum_k X[n][k] W[c][k] in fp32 for n < N, c < C (C = L*E stacked
// router rows): the router-logit contraction of Eq. 3 over calibration tokens.
int logits_gemm_launch(const uint16_t* X, int N, const uint16_t* W, int C, int d, float* H,
                       cudaStream_t stream) {
  using namespace gg;
  static PerDevice cache;
  const cudaError_t attr_err = static_cast<cudaError_t>(per_device(cache, [] {
    return static_cast<int>(cudaFuncSetAttribute(ffn_gemm_kernel<LOGITS>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 SMEM_BYTES));
  }));
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(logits)");
  CUtensorMap mX, mW;
  int rc;
  if ((rc = make_map(&mX, X, N, d))) return rc;
  if ((rc = make_map(&mW, W, C, d))) return rc;
  Args a{};
  a.offsets = nullptr;
  a.rows = N;
  a.n_valid = C;
  a.out_f32 = H;
  a.E = 1;
  a.K = d;
  a.n_tiles = (C + 255) / 256;
  a.b_rows = 0;
  a.limit_ns = wait_limit_ns();
  a.m_major = 1;  // the stacked router rows (a few MB) stay in L2; X_cal streams once
  const long long tiles = (long long)((N + BM - 1) / BM) * a.n_tiles;
  const int sms = num_sms();
  const int grid = static_cast<int>(tiles < sms ? tiles : sms);
  ffn_gemm_kernel<LOGITS><<<grid, THREADS, SMEM_BYTES, stream>>>(mX, mW, mW, a);
  OM_LAUNCHED("ffn_gemm_kernel<logits>");
  return ORDERMOE_OK;
}

// ---------------------------------------------------------- wait self-test
__global__ void wait_timeout_kernel(uint64_t limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // nothing ever arrives on `bar`: the wait must run out
    if (!mbar_wait(&bar, 0, limit_ns, reinterpret_cast<volatile int*>(&abort_flag)))
      report(&g_err_gemm, ORDERMOE_DEV_WAIT_TIMEOUT, 99);
  }
}

int selftest_wait_timeout(uint64_t limit_ns, cudaStream_t stream) {
  wait_timeout_kernel<<<1, 32, 0, stream>>>(limit_ns);
  OM_LAUNCHED("wait_timeout_kernel");
  return ORDERMOE_OK;
}

}  // namespace om

using namespace om;

static int ffn_check(const char* who, int R, int E, int d, int dff) {
  if (R < 0 || E <= 0 || E > ORDERMOE_MAX_EXPERTS)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "%s: need R >= 0 and 1 <= E <= 64", who);
  if (d <= 0 || d % 256 != 0 || dff <= 0 || dff % 128 != 0)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "%s: need d %% 256 == 0 and dff %% 128 == 0", who);
  if ((long long)E * dff > INT32_MAX || (long long)E * d > INT32_MAX || (long long)R * dff > INT32_MAX * 4LL)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "%s: sizes too large", who);
  return ORDERMOE_OK;
}

static bool all_aligned(std::initializer_list<const void*> ps) {
  for (const void* p : ps)
    if (!p || !aligned16(p)) return false;
  return true;
}

extern "C" int ordermoe_expert_ffn(const uint16_t* X_perm, const int32_t* offsets, int R,
                                   const uint16_t* W1, const uint16_t* W3, const uint16_t* W2,
                                   int E, int d, int dff, uint16_t* H, uint16_t* Y_perm,
                                   ordermoe_stream_t stream) {
  OM_TRACE();
  int rc = ffn_check("expert_ffn", R, E, d, dff);
  if (rc || R == 0) return rc;
  if (!offsets || !all_aligned({X_perm, W1, W3, W2, H, Y_perm}))
    return fail(ORDERMOE_ERR_INVALID_ARG, "expert_ffn: null or not 16-byte aligned pointer");
  return ffn_launch(X_perm, offsets, R, W1, W3, W2, E, d, dff, H, Y_perm, stream);
}

extern "C" int ordermoe_expert_gate_up(const uint16_t* X_perm, const int32_t* offsets, int R,
                                       const uint16_t* W1, const uint16_t* W3, int E, int d, int dff,
                                       uint16_t* H, ordermoe_stream_t stream) {
  OM_TRACE();
  int rc = ffn_check("expert_gate_up", R, E, d, dff);
  if (rc || R == 0) return rc;
  if (!offsets || !all_aligned({X_perm, W1, W3, H}))
    return fail(ORDERMOE_ERR_INVALID_ARG, "expert_gate_up: null or not 16-byte aligned pointer");
  return gate_up_launch(X_perm, offsets, R, W1, W3, E, d, dff, H, stream);
}

extern "C" int ordermoe_expert_down(const uint16_t* H, const int32_t* offsets, int R,
                                    const uint16_t* W2, int E, int d, int dff, uint16_t* Y_perm,
                                    ordermoe_stream_t stream) {
  OM_TRACE();
  int rc = ffn_check("expert_down", R, E, d, dff);
  if (rc || R == 0) return rc;
  if (!offsets || !all_aligned({H, W2, Y_perm}))
    return fail(ORDERMOE_ERR_INVALID_ARG, "expert_down: null or not 16-byte aligned pointer");
  return down_launch(H, offsets, R, W2, E, d, dff, Y_perm, stream);
}
