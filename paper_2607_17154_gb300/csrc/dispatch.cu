// Token permutation (histogram, prefix sum, stable scatter + row gather) and
// the weighted combine.
//
// Up to 4096 entries (a decode step) one block computes the histogram, the
// offsets and the stable ranks (dispatch_small_kernel). Otherwise the (token,
// slot) entries i = t*k + j are cut into chunks of kChunk = 256 consecutive
// entries, one block each:
//   1. chunk_hist: per-chunk expert histogram -> hist[E][chunk]
//   2. chunk_scan: one block; for every expert the exclusive prefix of its
//      count over chunks, plus the expert offsets (exclusive prefix over
//      experts) -> base[e][chunk] = offsets[e] + entries of e in earlier chunks
//   3. rank: stable rank inside the chunk (per-warp match + per-warp
//      counts), row = base + rank;
//   4. gather_rows: one warp per permuted row copies X[row_token[row]] into
//      X_perm with 16-byte loads and stores, over all SMs.
// Rows of one expert therefore keep the flat entry order: the permutation
// is unique and deterministic.
#include "common.cuh"

namespace om {

static __device__ unsigned long long g_err_dispatch = 0;

int read_clear_err_dispatch(unsigned long long* out) {
  unsigned long long zero = 0;
  OM_CUDA(cudaMemcpyFromSymbol(out, g_err_dispatch, sizeof(*out)));
  OM_CUDA(cudaMemcpyToSymbol(g_err_dispatch, &zero, sizeof(zero)));
  return ORDERMOE_OK;
}

constexpr int kChunk = kDispatchChunk;

__global__ void __launch_bounds__(kChunk) chunk_hist_kernel(const int32_t* __restrict__ chosen,
                                                            int64_t n, int E,
                                                            int32_t* __restrict__ hist) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  __shared__ int h[64];
  if (threadIdx.x < 64) h[threadIdx.x] = 0;
  __syncthreads();
  const int64_t i = (int64_t)blockIdx.x * kChunk + threadIdx.x;
  if (i < n) {
    const int e = chosen[i];
    if (e >= 0 && e < E) atomicAdd(&h[e], 1);
    else report(&g_err_dispatch, ORDERMOE_DEV_BAD_INDEX, static_cast<int>(i));
  }
  __syncthreads();
  if (threadIdx.x < E) hist[(size_t)threadIdx.x * gridDim.x + blockIdx.x] = h[threadIdx.x];
}

// One block of 1024 threads over hist[E][nchunks] (expert-major, as
// chunk_hist_kernel writes it): warp w scans the chunk counts of experts w
// and w + 32, then warp 0 scans the expert totals into offsets and they are
// added back: base[e][chunk] = offsets[e] + entries of e in earlier chunks.
// Up to kScanRegs * 32 chunks (T*k up to 65536 entries) both rows are loaded
// at once (coalesced: lane j holds chunks j, j + 32, ...) and scanned in
// registers, 32 chunks at a time with the running sum carried, and each base
// is written once. Longer rows go 32 chunks at a time from memory.
constexpr int kScanRegs = 8;

__device__ __forceinline__ int warp_excl_scan(int v, int lane, int* total) {
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += u;
  }
  *total = __shfl_sync(0xffffffffu, incl, 31);
  return incl - v;
}

__global__ void __launch_bounds__(1024, 1) chunk_scan_kernel(int32_t* __restrict__ hist, int nchunks,
                                                          int E, int32_t* __restrict__ offsets) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  __shared__ int total[64];
  __shared__ int start[65];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (nchunks <= 32 * kScanRegs) {
    int v[2][kScanRegs];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int e = warp + 32 * r;
#pragma unroll
      for (int i = 0; i < kScanRegs; ++i) {
        const int b = i * 32 + lane;
        v[r][i] = (e < E && b < nchunks) ? hist[(size_t)e * nchunks + b] : 0;
      }
    }
    int carry[2] = {0, 0};
#pragma unroll
    for (int i = 0; i < kScanRegs; ++i) {
      if (i * 32 < nchunks) {  // the same for the whole warp
#pragma unroll
        for (int r = 0; r < 2; ++r) {  // v becomes the row's exclusive prefix
          int sum;
          const int excl = warp_excl_scan(v[r][i], lane, &sum);
          v[r][i] = carry[r] + excl;
          carry[r] += sum;
        }
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r)
      if (lane == 0 && warp + 32 * r < E) total[warp + 32 * r] = carry[r];
    __syncthreads();
    if (warp == 0) {  // exclusive scan of the E <= 64 totals, two per lane
      const int t0 = (2 * lane < E) ? total[2 * lane] : 0;
      const int t1 = (2 * lane + 1 < E) ? total[2 * lane + 1] : 0;
      int all;
      const int excl = warp_excl_scan(t0 + t1, lane, &all);
      if (2 * lane < E) start[2 * lane] = excl;
      if (2 * lane + 1 < E) start[2 * lane + 1] = excl + t0;
      if (lane == 31) start[E] = all;
    }
    __syncthreads();
    if (threadIdx.x <= E) offsets[threadIdx.x] = start[threadIdx.x];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int e = warp + 32 * r;
      if (e >= E) continue;
      const int add = start[e];
#pragma unroll
      for (int i = 0; i < kScanRegs; ++i) {
        const int b = i * 32 + lane;
        if (b < nchunks) hist[(size_t)e * nchunks + b] = add + v[r][i];
      }
    }
    return;
  }
  for (int e = warp; e < E; e += 32) {
    int32_t* row = hist + (size_t)e * nchunks;
    int carry = 0;
    for (int b0 = 0; b0 < nchunks; b0 += 32) {
      const int b = b0 + lane;
      const int v = (b < nchunks) ? row[b] : 0;
      int incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += u;
      }
      if (b < nchunks) row[b] = carry + incl - v;
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) total[e] = carry;
  }
  __syncthreads();
  if (warp == 0) {  // exclusive scan of the E <= 64 totals, two per lane
    const int t0 = (2 * lane < E) ? total[2 * lane] : 0;
    const int t1 = (2 * lane + 1 < E) ? total[2 * lane + 1] : 0;
    int incl = t0 + t1;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int u = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += u;
    }
    const int excl = incl - t0 - t1;
    if (2 * lane < E) start[2 * lane] = excl;
    if (2 * lane + 1 < E) start[2 * lane + 1] = excl + t0;
    if (lane == 31) start[E] = incl;
  }
  __syncthreads();
  if (threadIdx.x <= E) offsets[threadIdx.x] = start[threadIdx.x];
  for (int e = warp; e < E; e += 32) {
    int32_t* row = hist + (size_t)e * nchunks;
    const int add = start[e];
    for (int b = lane; b < nchunks; b += 32) row[b] += add;
  }
}

__global__ void __launch_bounds__(kChunk) rank_kernel(
    const int32_t* __restrict__ chosen, int64_t n, int k, int E, const int32_t* __restrict__ base,
    int32_t* __restrict__ row_token, int32_t* __restrict__ row_of) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  constexpr int kWarps = kChunk / 32;
  __shared__ int cnt[kWarps][64];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < kWarps * 64; i += kChunk) (&cnt[0][0])[i] = 0;
  __syncthreads();
  const int64_t i = (int64_t)blockIdx.x * kChunk + threadIdx.x;
  const bool live = i < n;
  int e = live ? chosen[i] : -1;
  if (e >= E || e < -1) e = -1;  // reported by chunk_hist_kernel
  const unsigned peers = __match_any_sync(0xffffffffu, e);
  const int rank_in_warp = __popc(peers & ((1u << lane) - 1u));
  if (e >= 0 && rank_in_warp == 0) cnt[warp][e] = __popc(peers);
  __syncthreads();
  if (e >= 0) {
    int before = 0;
    for (int w = 0; w < warp; ++w) before += cnt[w][e];
    const int row = base[(size_t)e * gridDim.x + blockIdx.x] + before + rank_in_warp;
    row_of[i] = row;
    row_token[row] = static_cast<int32_t>(i / k);
  }
}

// X_perm[row] = X[row_token[row]]: one warp per row, kUnroll independent
// 16-byte loads per lane in flight, grid over all SMs.
// Only rows below offsets[E] were ranked (entries with a bad expert index are
// skipped and reported by chunk_hist_kernel).
__global__ void __launch_bounds__(256) gather_rows_kernel(const uint16_t* __restrict__ X,
                                                          const int32_t* __restrict__ row_token,
                                                          const int32_t* __restrict__ offsets,
                                                          int E, int T, int d,
                                                          uint16_t* __restrict__ X_perm) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  constexpr int kUnroll = 8;
  const int lane = threadIdx.x & 31;
  const int nvec = d >> 3;
  const int64_t R = offsets[E];
  const int64_t warps_total = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < R;
       r += warps_total) {
    const int64_t t = row_token[r];
    if (t < 0 || t >= T) {
      if (lane == 0) report(&g_err_dispatch, ORDERMOE_DEV_BAD_INDEX, static_cast<int>(r));
      continue;
    }
    const uint4* in = reinterpret_cast<const uint4*>(X + t * d);
    uint4* out = reinterpret_cast<uint4*>(X_perm + r * d);
    for (int v0 = lane; v0 < nvec; v0 += 32 * kUnroll) {
      uint4 buf[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int v = v0 + 32 * u;
        if (v < nvec) buf[u] = __ldg(in + v);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int v = v0 + 32 * u;
        if (v < nvec) out[v] = buf[u];
      }
    }
  }
}

// One warp per (token, part of 1024 columns): lane l handles the 16-byte
// vectors part * 128 + l + 32 u, u = 0..3, the loads of a slot in flight
// together; small batches (a decode step) still spread over many warps.
constexpr int kCombVec = 128;  // 16-byte vectors per warp item

__global__ void __launch_bounds__(256) combine_kernel(const uint16_t* __restrict__ Yp,
                                                      const int32_t* __restrict__ row_of,
                                                      const float* __restrict__ w, int T, int k,
                                                      int d, uint16_t* __restrict__ y) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t warps_total = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int nvec = d >> 3;
  const int parts = (nvec + kCombVec - 1) / kCombVec;
  const int64_t items = (int64_t)T * parts;
  for (int64_t it = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); it < items;
       it += warps_total) {
    const int t = static_cast<int>(it / parts);
    const int part = static_cast<int>(it - (int64_t)t * parts);
    // slot loops unrolled to the largest k with a j < k guard: constant indices keep
    // rows[] and ws[] in registers and let the loads of later slots issue early
    int rows[ORDERMOE_MAX_TOPK];
    float ws[ORDERMOE_MAX_TOPK];
    bool ok = true;
#pragma unroll
    for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j) {
      rows[j] = 0;
      ws[j] = 0.0f;
      if (j < k) {
        rows[j] = row_of[(size_t)t * k + j];
        ws[j] = w[(size_t)t * k + j];
        if (rows[j] < 0 || (int64_t)rows[j] >= (int64_t)T * k) ok = false;
      }
    }
    if (!ok) {  // a row index outside Y_perm: report, leave y[t] untouched
      if (lane == 0 && part == 0) report(&g_err_dispatch, ORDERMOE_DEV_BAD_INDEX, t);
      continue;
    }
    float acc[4][8];
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int x = 0; x < 8; ++x) acc[u][x] = 0.0f;
    const int v0 = part * kCombVec + lane;
#pragma unroll
    for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j) {
      if (j >= k) break;
      const uint4* src = reinterpret_cast<const uint4*>(Yp + (size_t)rows[j] * d);
      uint4 yv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (v0 + 32 * u < nvec) yv[u] = __ldg(src + v0 + 32 * u);
      const float wj = ws[j];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (v0 + 32 * u >= nvec) continue;
        acc[u][0] = fmaf(wj, bf16_lo(yv[u].x), acc[u][0]); acc[u][1] = fmaf(wj, bf16_hi(yv[u].x), acc[u][1]);
        acc[u][2] = fmaf(wj, bf16_lo(yv[u].y), acc[u][2]); acc[u][3] = fmaf(wj, bf16_hi(yv[u].y), acc[u][3]);
        acc[u][4] = fmaf(wj, bf16_lo(yv[u].z), acc[u][4]); acc[u][5] = fmaf(wj, bf16_hi(yv[u].z), acc[u][5]);
        acc[u][6] = fmaf(wj, bf16_lo(yv[u].w), acc[u][6]); acc[u][7] = fmaf(wj, bf16_hi(yv[u].w), acc[u][7]);
      }
    }
    uint4* dst = reinterpret_cast<uint4*>(y + (size_t)t * d);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (v0 + 32 * u >= nvec) continue;
      uint4 o;
      o.x = pack_bf16x2(acc[u][0], acc[u][1]); o.y = pack_bf16x2(acc[u][2], acc[u][3]);
      o.z = pack_bf16x2(acc[u][4], acc[u][5]); o.w = pack_bf16x2(acc[u][6], acc[u][7]);
      dst[v0 + 32 * u] = o;
    }
  }
}

// Pre-norm residual map between MoE layers (a decoder block without its
// attention half): h' = h + sum_j w_j Y_perm[row_of[t][j]] (the layer output
// added to the residual stream), x' = RMSNorm(h') = h' / sqrt(mean(h'^2) + eps)
// (the next layer's input, unit gain). One block of kNormThreads per token;
// thread i handles the 16-byte vectors i, i + kNormThreads, ...; the sum of
// squares is taken over the bf16 values written to h', reduced in a fixed
// order (warp butterflies, then the warps in order), so the result is
// deterministic. WITH_Y = false is RMSNorm alone (x = RMSNorm(h)).
constexpr int kNormThreads = 128;

template <bool WITH_Y>
__global__ void __launch_bounds__(kNormThreads) residual_norm_kernel(
    const uint16_t* __restrict__ Yp, const int32_t* __restrict__ row_of,
    const float* __restrict__ w, const uint16_t* __restrict__ h, int T, int k, int d, float eps,
    uint16_t* __restrict__ h_out, uint16_t* __restrict__ x_out) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  __shared__ float wsum[kNormThreads / 32];
  __shared__ int bad;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nvec = d >> 3;
  for (int t = blockIdx.x; t < T; t += gridDim.x) {
    int rows[ORDERMOE_MAX_TOPK];
    float ws[ORDERMOE_MAX_TOPK];
    if (tid == 0) bad = 0;
    __syncthreads();
#pragma unroll
    for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j) {
      rows[j] = 0;
      ws[j] = 0.0f;
      if (WITH_Y && j < k) {
        rows[j] = row_of[(size_t)t * k + j];
        ws[j] = w[(size_t)t * k + j];
        if (rows[j] < 0 || (int64_t)rows[j] >= (int64_t)T * k) bad = 1;
      }
    }
    __syncthreads();
    if (bad) {  // a row index outside Y_perm: report, leave token t untouched
      if (tid == 0) report(&g_err_dispatch, ORDERMOE_DEV_BAD_INDEX, t);
      __syncthreads();
      continue;
    }
    const uint4* hrow = reinterpret_cast<const uint4*>(h + (size_t)t * d);
    uint4* hw = reinterpret_cast<uint4*>(h_out + (size_t)t * d);
    float ss = 0.0f;
    for (int v = tid; v < nvec; v += kNormThreads) {
      const uint4 hv = __ldg(hrow + v);
      float a[8] = {bf16_lo(hv.x), bf16_hi(hv.x), bf16_lo(hv.y), bf16_hi(hv.y),
                    bf16_lo(hv.z), bf16_hi(hv.z), bf16_lo(hv.w), bf16_hi(hv.w)};
      if (WITH_Y) {
        uint4 yv[ORDERMOE_MAX_TOPK];
#pragma unroll
        for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j)
          if (j < k) yv[j] = __ldg(reinterpret_cast<const uint4*>(Yp + (size_t)rows[j] * d) + v);
#pragma unroll
        for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j) {
          if (j >= k) break;
          const float wj = ws[j];
          a[0] = fmaf(wj, bf16_lo(yv[j].x), a[0]); a[1] = fmaf(wj, bf16_hi(yv[j].x), a[1]);
          a[2] = fmaf(wj, bf16_lo(yv[j].y), a[2]); a[3] = fmaf(wj, bf16_hi(yv[j].y), a[3]);
          a[4] = fmaf(wj, bf16_lo(yv[j].z), a[4]); a[5] = fmaf(wj, bf16_hi(yv[j].z), a[5]);
          a[6] = fmaf(wj, bf16_lo(yv[j].w), a[6]); a[7] = fmaf(wj, bf16_hi(yv[j].w), a[7]);
        }
        uint4 o;
        o.x = pack_bf16x2(a[0], a[1]); o.y = pack_bf16x2(a[2], a[3]);
        o.z = pack_bf16x2(a[4], a[5]); o.w = pack_bf16x2(a[6], a[7]);
        hw[v] = o;
        const float r[8] = {bf16_lo(o.x), bf16_hi(o.x), bf16_lo(o.y), bf16_hi(o.y),
                            bf16_lo(o.z), bf16_hi(o.z), bf16_lo(o.w), bf16_hi(o.w)};
#pragma unroll
        for (int i = 0; i < 8; ++i) ss = fmaf(r[i], r[i], ss);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) ss = fmaf(a[i], a[i], ss);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if (lane == 0) wsum[warp] = ss;
    __syncthreads();
    float tot = 0.0f;
#pragma unroll
    for (int i = 0; i < kNormThreads / 32; ++i) tot += wsum[i];
    const float inv = __frsqrt_rn(__fadd_rn(__fdiv_rn(tot, static_cast<float>(d)), eps));
    // the residual values this thread wrote above (its own stores), or h
    const uint4* src = WITH_Y ? reinterpret_cast<const uint4*>(h_out + (size_t)t * d) : hrow;
    uint4* xw = reinterpret_cast<uint4*>(x_out + (size_t)t * d);
    for (int v = tid; v < nvec; v += kNormThreads) {
      const uint4 hv = src[v];
      uint4 o;
      o.x = pack_bf16x2(__fmul_rn(bf16_lo(hv.x), inv), __fmul_rn(bf16_hi(hv.x), inv));
      o.y = pack_bf16x2(__fmul_rn(bf16_lo(hv.y), inv), __fmul_rn(bf16_hi(hv.y), inv));
      o.z = pack_bf16x2(__fmul_rn(bf16_lo(hv.z), inv), __fmul_rn(bf16_hi(hv.z), inv));
      o.w = pack_bf16x2(__fmul_rn(bf16_lo(hv.w), inv), __fmul_rn(bf16_hi(hv.w), inv));
      xw[v] = o;
    }
    __syncthreads();  // wsum and bad are reused by the next token
  }
}

// Small batches (n <= kSmallN entries, e.g. a decode step): histogram, offsets
// and the stable rank in one block of 1024 threads. Pass 1 counts every
// expert; pass 2 walks the entries in rounds of 1024 in index order, ranks
// each round like rank_kernel and advances the experts' running starts, so
// the permutation equals the chunked path's.
constexpr int kSmallN = 4096;

__global__ void __launch_bounds__(1024) dispatch_small_kernel(
    const int32_t* __restrict__ chosen, int n, int k, int E, int32_t* __restrict__ offsets,
    int32_t* __restrict__ row_token, int32_t* __restrict__ row_of) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  __shared__ int total[64];
  __shared__ int start[64];
  __shared__ int wc[32][64];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid < 64) total[tid] = 0;
  __syncthreads();
  for (int i = tid; i < n; i += blockDim.x) {
    const int e = chosen[i];
    if (e >= 0 && e < E) atomicAdd(&total[e], 1);
    else report(&g_err_dispatch, ORDERMOE_DEV_BAD_INDEX, i);
  }
  __syncthreads();
  if (tid == 0) {
    int acc = 0;
    for (int x = 0; x < E; ++x) {
      start[x] = acc;
      offsets[x] = acc;
      acc += total[x];
    }
    offsets[E] = acc;
  }
  for (int r0 = 0; r0 < n; r0 += blockDim.x) {
    for (int x = tid; x < 32 * 64; x += blockDim.x) (&wc[0][0])[x] = 0;
    __syncthreads();
    const int i = r0 + tid;
    int e = i < n ? chosen[i] : -1;
    if (e >= E || e < -1) e = -1;  // reported in pass 1
    const unsigned peers = __match_any_sync(0xffffffffu, e);
    const int rank_in_warp = __popc(peers & ((1u << lane) - 1u));
    if (e >= 0 && rank_in_warp == 0) wc[warp][e] = __popc(peers);
    __syncthreads();
    if (e >= 0) {
      int before = 0;
      for (int w = 0; w < warp; ++w) before += wc[w][e];
      const int row = start[e] + before + rank_in_warp;
      row_of[i] = row;
      row_token[row] = i / k;
    }
    __syncthreads();
    if (tid < E) {
      int c = 0;
      for (int w = 0; w < 32; ++w) c += wc[w][tid];
      start[tid] += c;
    }
    __syncthreads();  // wc is read above before the next round clears it
  }
}

size_t dispatch_workspace_bytes(int64_t n, int E) {
  return (size_t)(dispatch_hist_entries(n, E) * sizeof(int32_t) + 255) & ~size_t(255);
}

int dispatch_launch(const int32_t* chosen, const uint16_t* X, int T, int k, int E, int d,
                    int32_t* offsets, int32_t* row_token, int32_t* row_of, uint16_t* X_perm,
                    int32_t* hist, cudaStream_t stream) {
  const int64_t n = (int64_t)T * k;
  const int nchunks = static_cast<int>((n + kChunk - 1) / kChunk);
  if (n == 0) {
    OM_CUDA(cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (E + 1), stream));
    return ORDERMOE_OK;
  }
  if (n <= kSmallN) {
    OM_LAUNCH_PDL("dispatch_small_kernel", dispatch_small_kernel, dim3(1), dim3(1024), 0, stream,
                  chosen, static_cast<int>(n), k, E, offsets, row_token, row_of);
  } else {
    OM_LAUNCH_PDL("chunk_hist_kernel", chunk_hist_kernel, dim3(nchunks), dim3(kChunk), 0, stream,
                  chosen, n, E, hist);
    OM_LAUNCH_PDL("chunk_scan_kernel", chunk_scan_kernel, dim3(1), dim3(1024), 0, stream,
                  hist, nchunks, E, offsets);
    OM_LAUNCH_PDL("rank_kernel", rank_kernel, dim3(nchunks), dim3(kChunk), 0, stream,
                  chosen, n, k, E, hist, row_token, row_of);
  }
  int64_t blocks = (n + 7) / 8;
  const int cap = num_sms() * 8;
  if (blocks > cap) blocks = cap;
  OM_LAUNCH_PDL("gather_rows_kernel", gather_rows_kernel, dim3(static_cast<int>(blocks)), dim3(256),
                0, stream, X, row_token, offsets, E, T, d, X_perm);
  return ORDERMOE_OK;
}

}  // namespace om

using namespace om;

extern "C" size_t ordermoe_dispatch_workspace_bytes(int T, int k, int E) {
  if (T < 0 || k <= 0 || E <= 0 || E > ORDERMOE_MAX_EXPERTS) return 0;
  return om::dispatch_workspace_bytes((int64_t)T * k, E);
}

extern "C" int ordermoe_dispatch(const int32_t* chosen_expert, const uint16_t* X, int T, int k,
                                 int E, int d, int32_t* offsets, int32_t* row_token,
                                 int32_t* row_of, uint16_t* X_perm, void* workspace,
                                 size_t workspace_bytes, ordermoe_stream_t stream) {
  OM_TRACE();
  if (T < 0 || k <= 0 || k > ORDERMOE_MAX_TOPK || E <= 0 || E > ORDERMOE_MAX_EXPERTS)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "dispatch: need T >= 0, 1 <= k <= 8, 1 <= E <= 64");
  if (d <= 0 || d % 8 != 0)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "dispatch: d must be a positive multiple of 8");
  if (!offsets) return fail(ORDERMOE_ERR_INVALID_ARG, "dispatch: null offsets");
  if (T > 0 && (!chosen_expert || !X || !row_token || !row_of || !X_perm || !workspace))
    return fail(ORDERMOE_ERR_INVALID_ARG, "dispatch: null pointer");
  if ((int64_t)T * k > INT32_MAX) return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "dispatch: T*k too large");
  if (T > 0 && (!aligned16(X) || !aligned16(X_perm)))
    return fail(ORDERMOE_ERR_INVALID_ARG, "dispatch: X and X_perm must be 16-byte aligned");
  if (workspace_bytes < om::dispatch_workspace_bytes((int64_t)T * k, E))
    return fail(ORDERMOE_ERR_INVALID_ARG, "dispatch: workspace too small");
  return dispatch_launch(chosen_expert, X, T, k, E, d, offsets, row_token, row_of, X_perm,
                         static_cast<int32_t*>(workspace), stream);
}

static bool overlaps(const void* a, const void* b, size_t bytes) {
  const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
  return x < y + bytes && y < x + bytes;
}

extern "C" int ordermoe_rmsnorm(const uint16_t* h, int T, int d, float eps, uint16_t* x,
                                ordermoe_stream_t stream) {
  OM_TRACE();
  if (T < 0 || d <= 0 || d % 8 != 0)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "rmsnorm: need T >= 0 and d a positive multiple of 8");
  if (!(eps > 0.0f)) return fail(ORDERMOE_ERR_INVALID_ARG, "rmsnorm: eps must be > 0");
  if (T == 0) return ORDERMOE_OK;
  if (!h || !x || !aligned16(h) || !aligned16(x))
    return fail(ORDERMOE_ERR_INVALID_ARG, "rmsnorm: null or not 16-byte aligned pointer");
  const int grid = T < num_sms() * 16 ? T : num_sms() * 16;
  OM_LAUNCH_PDL("residual_norm_kernel<rmsnorm>", residual_norm_kernel<false>, dim3(grid),
                dim3(kNormThreads), 0, stream, nullptr, nullptr, nullptr, h, T, 1, d, eps, nullptr,
                x);
  return ORDERMOE_OK;
}

extern "C" int ordermoe_combine_residual_norm(const uint16_t* Y_perm, const int32_t* row_of,
                                              const float* topk_w, const uint16_t* h, int T, int k,
                                              int d, float eps, uint16_t* h_out, uint16_t* x_out,
                                              ordermoe_stream_t stream) {
  OM_TRACE();
  if (T < 0 || k <= 0 || k > ORDERMOE_MAX_TOPK)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "combine_residual_norm: need T >= 0, 1 <= k <= 8");
  if (d <= 0 || d % 8 != 0)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE,
                "combine_residual_norm: d must be a positive multiple of 8");
  if (!(eps > 0.0f)) return fail(ORDERMOE_ERR_INVALID_ARG, "combine_residual_norm: eps must be > 0");
  if (T == 0) return ORDERMOE_OK;
  if (!Y_perm || !row_of || !topk_w || !h || !h_out || !x_out)
    return fail(ORDERMOE_ERR_INVALID_ARG, "combine_residual_norm: null pointer");
  if (!aligned16(Y_perm) || !aligned16(h) || !aligned16(h_out) || !aligned16(x_out))
    return fail(ORDERMOE_ERR_INVALID_ARG, "combine_residual_norm: bf16 arrays must be 16-byte aligned");
  const size_t row_bytes = (size_t)T * d * 2;
  if (overlaps(h, h_out, row_bytes) || overlaps(h, x_out, row_bytes) ||
      overlaps(h_out, x_out, row_bytes))
    return fail(ORDERMOE_ERR_INVALID_ARG, "combine_residual_norm: h, h_out and x_out must not overlap");
  const int grid = T < num_sms() * 16 ? T : num_sms() * 16;
  OM_LAUNCH_PDL("residual_norm_kernel<combine>", residual_norm_kernel<true>, dim3(grid),
                dim3(kNormThreads), 0, stream, Y_perm, row_of, topk_w, h, T, k, d, eps, h_out, x_out);
  return ORDERMOE_OK;
}

extern "C" int ordermoe_combine(const uint16_t* Y_perm, const int32_t* row_of,
                                const float* topk_w, int T, int k, int d, uint16_t* y,
                                ordermoe_stream_t stream) {
  OM_TRACE();
  if (T < 0 || k <= 0 || k > ORDERMOE_MAX_TOPK)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "combine: need T >= 0, 1 <= k <= 8");
  if (d <= 0 || d % 8 != 0)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "combine: d must be a positive multiple of 8");
  if (T == 0) return ORDERMOE_OK;
  if (!Y_perm || !row_of || !topk_w || !y) return fail(ORDERMOE_ERR_INVALID_ARG, "combine: null pointer");
  if (!aligned16(Y_perm) || !aligned16(y))
    return fail(ORDERMOE_ERR_INVALID_ARG, "combine: Y_perm and y must be 16-byte aligned");
  const int64_t items = (int64_t)T * (((d >> 3) + kCombVec - 1) / kCombVec);
  int64_t blocks = (items + 7) / 8;  // 8 warps per block
  const int cap = num_sms() * 8;
  if (blocks > cap) blocks = cap;
  OM_LAUNCH_PDL("combine_kernel", combine_kernel, dim3(static_cast<int>(blocks)), dim3(256), 0,
                stream, Y_perm, row_of, topk_w, T, k, d, y);
  return ORDERMOE_OK;
}
