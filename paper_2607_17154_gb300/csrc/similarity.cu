// Offline planning on the GPU (Section IV, Alg. 1 grouping and placement):
//   ordermoe_similarity: H = W_r X_cal^T (Eq. 3, tcgen05 GEMM into scratch),
//     Sim = cosine of the rows of H (Eq. 4), activation counts n_j (Eq. 5);
//   ordermoe_expert_counts: the counts of Eq. 5 from given logits;
//   ordermoe_place: threshold (Eq. 6), greedy grouping (Eqs. 24-26),
//     importance (Eqs. 27-28) and mandatory placement (Eqs. 29-31);
//   ordermoe_replicate: redundant deployment (Eqs. 32-35);
//   ordermoe_coverage: local group coverage (Eq. 32).
#include "common.cuh"

namespace om {

int logits_gemm_launch(const uint16_t* X, int N, const uint16_t* W, int C, int d, float* H,
                       cudaStream_t stream);

static __device__ unsigned long long g_err_sim = 0;

int read_clear_err_sim(unsigned long long* out) {
  unsigned long long zero = 0;
  OM_CUDA(cudaMemcpyFromSymbol(out, g_err_sim, sizeof(*out)));
  OM_CUDA(cudaMemcpyToSymbol(g_err_sim, &zero, sizeof(zero)));
  return ORDERMOE_OK;
}

constexpr int kSimChunk = 1024;  // calibration tokens per partial Gram
constexpr int kSub = 64;         // tokens staged in shared memory at a time

// Rank order used for top-k: larger logit first, equal logits by lower index.
__device__ __forceinline__ void add_topk_counts(const float* l, int E, int kf, int* counts) {
  unsigned long long used = 0;
  for (int j = 0; j < kf; ++j) {
    int best = -1;
    float bv = 0.0f;
    for (int e = 0; e < E; ++e) {
      if ((used >> e) & 1ull) continue;
      if (best < 0 || l[e] > bv) { best = e; bv = l[e]; }
    }
    used |= 1ull << best;
    atomicAdd(&counts[best], 1);
  }
}

// grid (chunks, L), 256 threads. Partial Gram of layer l over one chunk of
// tokens: thread (ti, tj) of a 16 x 16 grid accumulates the 4 x 4 block
// G[4 ti .. 4 ti + 3][4 tj .. 4 tj + 3] in fp32; each staged token costs two
// float4 shared loads per 16 FMAs.
__global__ void __launch_bounds__(256) gram_kernel(const float* __restrict__ H, int64_t N, int L,
                                                   int E, float* __restrict__ gpart) {
  __shared__ __align__(16) float sh[kSub][64];
  // the layers of one chunk are neighbouring blocks, so each token's record
  // of L * E logits is read from DRAM once and shared through L2
  const int l = blockIdx.x, chunk = blockIdx.y;
  const int nchunks = gridDim.y;
  const int tid = threadIdx.x;
  const int ti = tid >> 4, tj = tid & 15;
  const int LE = L * E;
  float acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.0f;
  const int64_t n_begin = (int64_t)chunk * kSimChunk;
  int64_t n_end = n_begin + kSimChunk;
  if (n_end > N) n_end = N;
  const bool active = 4 * ti < E && 4 * tj < E;
  for (int64_t n0 = n_begin; n0 < n_end; n0 += kSub) {
    __syncthreads();
    if ((E & 3) == 0 && (LE & 3) == 0) {
      // 16 float4 per token row; each thread stages 4 of the 1024 float4
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int x = tid + 256 * u;
        const int r = x >> 4, c4 = (x & 15) * 4;
        const int64_t n = n0 + r;
        float4 v = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        if (n < n_end && c4 < E)
          v = *reinterpret_cast<const float4*>(H + n * LE + (int64_t)l * E + c4);
        *reinterpret_cast<float4*>(&sh[r][c4]) = v;
      }
    } else {
      for (int x = tid; x < kSub * 64; x += 256) {
        const int r = x >> 6, c = x & 63;
        const int64_t n = n0 + r;
        sh[r][c] = (n < n_end && c < E) ? H[n * LE + (int64_t)l * E + c] : 0.0f;
      }
    }
    __syncthreads();
    if (active) {
#pragma unroll 4
      for (int r = 0; r < kSub; ++r) {
        const float4 a = *reinterpret_cast<const float4*>(&sh[r][4 * ti]);
        const float4 b = *reinterpret_cast<const float4*>(&sh[r][4 * tj]);
#define OM_GRAM_ROW(p, ap)                       \
  acc[p][0] = fmaf(ap, b.x, acc[p][0]);          \
  acc[p][1] = fmaf(ap, b.y, acc[p][1]);          \
  acc[p][2] = fmaf(ap, b.z, acc[p][2]);          \
  acc[p][3] = fmaf(ap, b.w, acc[p][3]);
        OM_GRAM_ROW(0, a.x) OM_GRAM_ROW(1, a.y) OM_GRAM_ROW(2, a.z) OM_GRAM_ROW(3, a.w)
#undef OM_GRAM_ROW
      }
    }
  }
  float* gp = gpart + ((size_t)l * nchunks + chunk) * 64 * 64;
  if (active)
#pragma unroll
    for (int p = 0; p < 4; ++p)
#pragma unroll
      for (int q = 0; q < 4; ++q) gp[(4 * ti + p) * 64 + 4 * tj + q] = acc[p][q];
}

// Eq. 5 counts from the token-major logits H[n][l E + e]: one thread per
// (token, layer) holds the layer's E logits in registers and takes k_freq
// passes (larger logit first, lower index on ties). Block totals are added
// with integer atomics, so the result does not depend on the order.
template <int EMAX>
__global__ void __launch_bounds__(256) counts_kernel(const float* __restrict__ H, int64_t N, int L,
                                                     int E, int kf, int32_t* __restrict__ counts) {
  __shared__ int cnt[64];
  const int l = blockIdx.x;  // layers of the same tokens run side by side (L2 reuse)
  if (threadIdx.x < 64) cnt[threadIdx.x] = 0;
  __syncthreads();
  const int LE = L * E;
  const bool vec = (E & 3) == 0 && (LE & 3) == 0;
  for (int64_t n = (int64_t)blockIdx.y * blockDim.x + threadIdx.x; n < N;
       n += (int64_t)gridDim.y * blockDim.x) {
    const float* row = H + n * LE + (int64_t)l * E;
    float v[EMAX];
    if (vec) {
#pragma unroll
      for (int e = 0; e < EMAX; e += 4) {
        if (e < E) {
          const float4 q = *reinterpret_cast<const float4*>(row + e);
          v[e] = q.x; v[e + 1] = q.y; v[e + 2] = q.z; v[e + 3] = q.w;
        }
      }
    } else {
#pragma unroll
      for (int e = 0; e < EMAX; ++e)
        if (e < E) v[e] = row[e];
    }
    unsigned long long used = 0;
    for (int j = 0; j < kf; ++j) {
      int best = -1;
      float bv = 0.0f;
#pragma unroll
      for (int e = 0; e < EMAX; ++e) {
        if (e < E && !((used >> e) & 1ull) && (best < 0 || v[e] > bv)) {
          best = e;
          bv = v[e];
        }
      }
      used |= 1ull << best;
      atomicAdd(&cnt[best], 1);
    }
  }
  __syncthreads();
  if (threadIdx.x < E && cnt[threadIdx.x]) atomicAdd(&counts[(size_t)l * E + threadIdx.x], cnt[threadIdx.x]);
}

// Top-kf of one token's E logits (rank order: larger first, lower index on
// ties) as a bit set.
template <int EMAX>
__device__ __forceinline__ unsigned long long topk_set(const float* __restrict__ row, int E, int kf) {
  float v[EMAX];
#pragma unroll
  for (int e = 0; e < EMAX; ++e) v[e] = (e < E) ? row[e] : 0.0f;
  unsigned long long used = 0;
  for (int j = 0; j < kf; ++j) {
    int best = -1;
    float bv = 0.0f;
#pragma unroll
    for (int e = 0; e < EMAX; ++e)
      if (e < E && !((used >> e) & 1ull) && (best < 0 || v[e] > bv)) {
        best = e;
        bv = v[e];
      }
    used |= 1ull << best;
  }
  return used;
}

// Transition counts of Eq. 41 for the layer pair (l, l + 1) = blockIdx.y:
// each token adds one to n_l(k -> k') for every k in its top-kf at layer l
// and k' in its top-kf at layer l + 1 (integer atomics: order-independent).
template <int EMAX>
// logits of token n at layer l start at n * sn + l * sl (floats).
__global__ void __launch_bounds__(256) transitions_kernel(const float* __restrict__ logits,
                                                          int64_t N, int L, int E, int kf,
                                                          int64_t sn, int64_t sl,
                                                          int32_t* __restrict__ counts) {
  __shared__ int h[64 * 64];
  const int l = blockIdx.y;
  for (int i = threadIdx.x; i < E * E; i += blockDim.x) h[i] = 0;
  __syncthreads();
  for (int64_t n = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; n < N;
       n += (int64_t)gridDim.x * blockDim.x) {
    unsigned long long a = topk_set<EMAX>(logits + n * sn + l * sl, E, kf);
    const unsigned long long b = topk_set<EMAX>(logits + n * sn + (l + 1) * sl, E, kf);
    while (a) {
      const int x = __ffsll(static_cast<long long>(a)) - 1;
      a &= a - 1;
      unsigned long long bb = b;
      while (bb) {
        const int y = __ffsll(static_cast<long long>(bb)) - 1;
        bb &= bb - 1;
        atomicAdd(&h[x * E + y], 1);
      }
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < E * E; i += blockDim.x)
    if (h[i]) atomicAdd(&counts[(size_t)l * E * E + i], h[i]);
}

// P_l(k -> k') = n / sum_k'' n (fp64, rounded once to fp32); 0 for an empty row.
__global__ void transitions_finish_kernel(const int32_t* __restrict__ counts, int rows, int E,
                                          float* __restrict__ P) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= rows) return;
  const int32_t* c = counts + (size_t)r * E;
  double row = 0.0;
  for (int b = 0; b < E; ++b) row = __dadd_rn(row, static_cast<double>(c[b]));
  for (int b = 0; b < E; ++b)
    P[(size_t)r * E + b] = row > 0.0 ? __double2float_rn(__ddiv_rn(static_cast<double>(c[b]), row)) : 0.0f;
}

// grid (L, 16), 256 threads: block (l, b) reduces the 256 Gram entries
// i * 64 + j in [256 b, 256 b + 256) over the chunks, in chunk order (fp64).
__global__ void __launch_bounds__(256) gram_reduce_kernel(const float* __restrict__ gpart,
                                                          int nchunks, double* __restrict__ G) {
  const int l = blockIdx.x;
  const int x = blockIdx.y * 256 + threadIdx.x;
  const float* src = gpart + (size_t)l * nchunks * 4096 + x;
  double s = 0.0;
  int c = 0;
  for (; c + 8 <= nchunks; c += 8) {
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = src[(size_t)(c + u) * 4096];
#pragma unroll
    for (int u = 0; u < 8; ++u) s += static_cast<double>(v[u]);
  }
  for (; c < nchunks; ++c) s += static_cast<double>(src[(size_t)c * 4096]);
  G[(size_t)l * 4096 + x] = s;
}

// grid (L, 16): Sim(i,j) = G_ij / (sqrt(G_ii) sqrt(G_jj)) (Eq. 4), diagonal 1,
// zero-norm 0; block y takes entries 256 y .. 256 y + 255 of layer l (the fp64
// square roots and divides of a layer spread over 16 SMs).
__global__ void __launch_bounds__(256) sim_finish_kernel(const double* __restrict__ Gall, int E,
                                                         float* __restrict__ sim) {
  __shared__ double norm[64];
  const int l = blockIdx.x;
  const double* G = Gall + (size_t)l * 4096;
  if (threadIdx.x < E) norm[threadIdx.x] = sqrt(G[threadIdx.x * 64 + threadIdx.x]);
  __syncthreads();
  const int x = blockIdx.y * 256 + threadIdx.x;
  if (x >= E * E) return;
  const int i = x / E, j = x % E;
  float v;
  if (i == j) {
    v = 1.0f;
  } else {
    const double ni = norm[i], nj = norm[j];
    v = (ni == 0.0 || nj == 0.0) ? 0.0f : __double2float_rn(G[i * 64 + j] / (ni * nj));
  }
  sim[(size_t)l * E * E + x] = v;
}

__global__ void counts_from_logits_kernel(const float* __restrict__ logits, int64_t N, int E,
                                          int kf, int32_t* __restrict__ counts) {
  __shared__ int cnt[64];
  if (threadIdx.x < 64) cnt[threadIdx.x] = 0;
  __syncthreads();
  for (int64_t n = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; n < N;
       n += (int64_t)gridDim.x * blockDim.x) {
    float l[64];
    for (int e = 0; e < E; ++e) l[e] = logits[n * E + e];
    add_topk_counts(l, E, kf, cnt);
  }
  __syncthreads();
  if (threadIdx.x < E && cnt[threadIdx.x]) atomicAdd(&counts[threadIdx.x], cnt[threadIdx.x]);
}

// ---------------------------------------------------------------------------
// Grouping and placement: one block of 64 threads, layers in order. Thread e
// owns expert e in the parallel parts; the greedy loops are sequential in the
// paper's order. fp64 arithmetic uses explicit round-to-nearest operations.
struct PlaceParams {
  double theta_min, theta_max, theta_single;
  double alpha_f, alpha_r, lambda1, lambda2;
};

// Integer key of an fp64 value for a descending order with NaN after every
// number: larger values get larger keys (the bits, sign-flipped for
// negatives, with -0 taken as +0), and every NaN gets 0, below them all.
__device__ __forceinline__ unsigned long long rank_key(double x) {
  if (x != x) return 0ull;
  unsigned long long b = static_cast<unsigned long long>(__double_as_longlong(x == 0.0 ? 0.0 : x));
  return (b >> 63) ? ~b : (b | 0x8000000000000000ull);
}

// One layer's scratch of the grouping.
struct GroupSmem {
  unsigned long long kp[64];  // rank_key of p and of I, for the placement order
  unsigned long long ki[64];
  double imp[64];
  double pls[64];
  int order[64];
  int dom[64];
  int grp[64];
  int cnt[64];
  float S[64 * 64];
};

// Per-layer part of the plan for layer l, on 64 threads t = 0..63 of a block
// (the layers are independent here): theta_l (Eq. 6), greedy cover
// (Eqs. 24-26), importance (Eqs. 27-28) and the placement order (p desc,
// I desc, index asc). A slice with live == false has no layer this round but
// meets every barrier of the block.
__device__ void group_layer(GroupSmem& sm, bool live, int t, int l, const float* __restrict__ sim,
                            const int32_t* __restrict__ counts, int L, int E, PlaceParams pp,
                            const double* __restrict__ p, int32_t* __restrict__ group,
                            int32_t* __restrict__ n_groups, float* __restrict__ theta_out,
                            double* __restrict__ importance, int32_t* __restrict__ porder) {
  double* imp = sm.imp;
  double* pls = sm.pls;
  int* order = sm.order;
  int* dom = sm.dom;
  int* grp = sm.grp;
  int* cnt = sm.cnt;
  float* S = sm.S;
  if (live) {
    for (int i = t; i < E * E; i += 64) S[i] = sim[(size_t)l * E * E + i];
    if (t < E) {
      cnt[t] = counts[(size_t)l * E + t];
      pls[t] = p[(size_t)l * E + t];
      if (!(pls[t] >= 0.0)) report(&g_err_sim, ORDERMOE_DEV_BAD_VALUE, l * E + t);  // Eq. 29's p
    }
  }
  __syncthreads();
  // Eq. 6 (layers numbered from 1)
  float theta;
  if (L <= 1) {
    theta = __double2float_rn(pp.theta_single);
  } else {
    const double frac = __ddiv_rn(static_cast<double>(L - (l + 1)), static_cast<double>(L - 1));
    theta = __double2float_rn(
        __dadd_rn(pp.theta_min, __dmul_rn(__dsub_rn(pp.theta_max, pp.theta_min), frac)));
  }
  // visiting order: count desc, index asc
  if (live && t < E) {
    int r = 0;
    for (int e = 0; e < E; ++e)
      if (cnt[e] > cnt[t] || (cnt[e] == cnt[t] && e < t)) ++r;
    order[r] = t;
  }
  __syncthreads();
  // Eqs. 24-26 in the visiting order; warp 0 scans the existing dominants in
  // parallel (lane g takes dominants g and g + 32; ties to the earlier one).
  // The choice is the scan's in dominant order: the first dominant unless a
  // later one is strictly more similar. With NaN similarities that is the
  // first dominant when its similarity is NaN, else the first maximum with
  // NaN counted as -inf: a total order, so every lane of the reduction ends
  // with the same group.
  if (live && t < 32) {
    int k = 0;
    for (int pos = 0; pos < E; ++pos) {
      const int j = order[pos];
      float bs = -INFINITY;
      int bg = 1 << 30;
      for (int g = t; g < k; g += 32) {
        const float sv = S[j * E + dom[g]];
        const float v = sv != sv ? -INFINITY : sv;
        if (bg == (1 << 30) || v > bs) { bg = g; bs = v; }
      }
      // across the lanes: the largest similarity by an order-preserving 32-bit
      // key (0: the lane has no dominant; -0 counted as +0, so that equal
      // similarities are equal keys), then the lowest dominant index among
      // the lanes that hold it (dominants below 32 before those above)
      uint32_t key = 0u;
      if (bg != (1 << 30)) {
        const uint32_t u = __float_as_uint(bs == 0.0f ? 0.0f : bs);
        key = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
      }
      const uint32_t mk = __reduce_max_sync(0xffffffffu, key);
      const unsigned lo32 = __ballot_sync(0xffffffffu, key == mk && bg < 32);
      const unsigned hi32 = __ballot_sync(0xffffffffu, key == mk && bg >= 32 && bg != (1 << 30));
      if (mk == 0u) {
        bg = 1 << 30;
      } else {
        bg = lo32 ? __ffs(lo32) - 1 : __ffs(hi32) - 1 + 32;
        bs = __uint_as_float((mk & 0x80000000u) ? (mk & 0x7FFFFFFFu) : ~mk);
      }
      if (k > 0) {
        const float s0 = S[j * E + dom[0]];
        if (s0 != s0) {  // NaN first: the scan keeps dominant 0 (and NaN < theta is false)
          bg = 0;
          bs = s0;
        }
      }
      if (bg == (1 << 30) || bs < theta) {
        if (t == 0) { dom[k] = j; grp[j] = k; }
        ++k;
      } else if (t == 0) {
        grp[j] = bg;
      }
      __syncwarp();
    }
    if (t == 0) {
      n_groups[l] = k;
      theta_out[l] = theta;
    }
  }
  __syncthreads();
  // Eqs. 27-28
  // the counts' fp64 sum in index order, formed exactly as an integer sum
  // (every partial sum is an integer below 2^53, so each fp64 addition is exact)
  long long total_i = 0;
  if (live)
    for (int e = 0; e < E; ++e) total_i += cnt[e];
  const double total = static_cast<double>(total_i);
  if (live && t < E) {
    group[(size_t)l * E + t] = grp[t];
    double sum = 0.0;
    int size = 0;
    for (int k2 = 0; k2 < E; ++k2)
      if (grp[k2] == grp[t]) { sum = __dadd_rn(sum, static_cast<double>(S[t * E + k2])); ++size; }
    const double rho = __ddiv_rn(sum, static_cast<double>(size));
    const double f = total > 0.0 ? __ddiv_rn(static_cast<double>(cnt[t]), total) : 0.0;
    imp[t] = __dadd_rn(__dmul_rn(pp.alpha_f, f), __dmul_rn(pp.alpha_r, rho));
    if (importance != nullptr) importance[(size_t)l * E + t] = imp[t];
  }
  __syncthreads();
  // placement order: p desc, I desc, index asc, with NaN after every number
  // (a total order, so the ranks are a permutation whatever the values),
  // compared on integer keys
  if (live && t < E) {
    sm.kp[t] = rank_key(pls[t]);
    sm.ki[t] = rank_key(imp[t]);
  }
  __syncthreads();
  if (live && t < E) {
    const unsigned long long kpt = sm.kp[t], kit = sm.ki[t];
    int r = 0;
    for (int e = 0; e < E; ++e) {
      const unsigned long long kpe = sm.kp[e], kie = sm.ki[e];
      r += (kpe > kpt || (kpe == kpt && (kie > kit || (kie == kit && e < t)))) ? 1 : 0;
    }
    porder[(size_t)l * E + r] = t;
  }
}

// One block per layer l = l0 + blockIdx.x, 64 threads.
__global__ void __launch_bounds__(64) group_kernel(
    const float* __restrict__ sim, const int32_t* __restrict__ counts, int L, int E, int l0,
    PlaceParams pp, const double* __restrict__ p, int32_t* __restrict__ group,
    int32_t* __restrict__ n_groups, float* __restrict__ theta_out, double* __restrict__ importance,
    int32_t* __restrict__ porder) {
  __shared__ GroupSmem sm;
  group_layer(sm, true, threadIdx.x, l0 + blockIdx.x, sim, counts, L, E, pp, p, group, n_groups,
              theta_out, importance, porder);
}

// b / C rounded to nearest by Markstein's correction step (P. Markstein, IBM J.
// Res. Dev. 34(1), 1990): with y = 1/C rounded to nearest and q = RN(b y)
// within one ulp of b / C, the residual r = b - C q is exact in one fma, and
// RN(q + r y) is the correctly rounded quotient (no underflow or overflow).
// Three dependent fp64 operations instead of a full division.
__device__ __forceinline__ double div_rn_markstein(double b, double C, double y) {
  const double q = __dmul_rn(b, y);
  const double r = __fma_rn(-q, C, b);
  return __fma_rn(r, y, q);
}

__global__ void div_selftest_kernel(const double* __restrict__ a, const double* __restrict__ b,
                                    double* __restrict__ out, int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    out[i] = div_rn_markstein(a[i], b[i], __drcp_rn(b[i]));
}

// Mandatory placement, Eqs. 29-31 (Alg. 1): one warp, layers and
// experts in order, b_m carried over the layers. Lane m keeps server m's
// state in registers: b_m, C_m and lambda1 * (b_m / C_m); lambda2 * eta for
// every count is a table. Per expert, lane m forms its score (one fp64 add of
// the two terms, as Eq. 30 states them) and, speculatively, the ratio term it
// would have after taking the expert; the argmin runs on integer keys
// (scores are non-negative, so their bit patterns order like the values; ties
// to the lower server), and the winner keeps its speculative term. A
// waiting-list expert goes to the server with the most room after its layer.
// Layers l0 .. l1 - 1: the first range starts from b_m = 0 and sets the
// status, a later range continues from b_m in used (lambda1 * (b_m / C_m) is
// recomputed from it, the same function the loop applies) and only raises the
// capacity status.
struct PlaceSmem {
  int grp[64];
  int ord[64];
  double pls[64];
  int waiting[64];
  uint8_t xs[32 * 64];
  int eta[32 * 64];
  double l2eta[65];  // lambda2 * eta for eta = 0 .. 64
};

// The placement on warp 0 of a block (threadIdx.x < 32); returns 1 when a
// waiting-list expert overfilled its server.
__device__ int place_layers(PlaceSmem& sm, const int32_t* __restrict__ group,
                             const int32_t* __restrict__ porder, int L, int E, int M, int l0,
                             int l1, int first, PlaceParams pp, const double* __restrict__ p,
                             const double* __restrict__ C, uint8_t* __restrict__ placement,
                             double* __restrict__ used) {
  int* grp = sm.grp;
  int* ord = sm.ord;
  double* pls = sm.pls;
  int* waiting = sm.waiting;
  uint8_t* xs = sm.xs;
  int* eta = sm.eta;
  double* l2eta = sm.l2eta;
  const int t = threadIdx.x;
  int overflow = 0;
  const bool srv = t < M;
  double b = (srv && !first) ? used[t] : 0.0;
  const double cap = srv ? C[t] : 1.0;
  const double rcap = __drcp_rn(cap);
  // non-negative finite values compare like their bit patterns
  const long long cap_bits = __double_as_longlong(cap);
  double a1 = srv ? __dmul_rn(pp.lambda1, div_rn_markstein(b, cap, rcap)) : 0.0;
  bool bad_score = srv && !(cap > 0.0 && cap <= 1.7976931348623157e308);
  for (int i = t; i <= 64; i += 32) l2eta[i] = __dmul_rn(pp.lambda2, static_cast<double>(i));
  __syncwarp();
  for (int l = l0; l < l1; ++l) {
    for (int i = t; i < 32 * 64; i += 32) {
      xs[i] = 0;
      eta[i] = 0;
    }
    for (int e = t; e < E; e += 32) {
      grp[e] = group[(size_t)l * E + e];
      ord[e] = porder[(size_t)l * E + e];
      pls[e] = p[(size_t)l * E + e];
    }
    __syncwarp();
    int nw = 0;
    int jn = ord[0];
    int gn = grp[jn];
    double pn = pls[jn];
    for (int pos = 0; pos < E; ++pos) {
      const int j = jn, g = gn;
      const double pj = pn;
      if (pos + 1 < E) {  // the next expert does not depend on this one's outcome
        jn = ord[pos + 1];
        gn = grp[jn];
        pn = pls[jn];
      }
      // the fp64 work on the server lanes only (the other lanes' keys are ~0)
      double bn = 0.0, a1n = 0.0;
      unsigned long long key = ~0ull;
      if (srv) {
        bn = __dadd_rn(b, pj);
        const bool feas = __double_as_longlong(bn) <= cap_bits;  // bn <= C_m, bn >= 0
        const int et = min(eta[t * 64 + g], 64);  // at most E <= 64
        const double sc = __dadd_rn(a1, l2eta[et]);
        if (feas) {
          a1n = __dmul_rn(pp.lambda1, div_rn_markstein(bn, cap, rcap));  // kept if this lane wins
          unsigned long long ks = static_cast<unsigned long long>(__double_as_longlong(sc));
          // !(sc >= 0) on the bits: a NaN, or a negative value other than -0
          const unsigned long long mag = ks & 0x7FFFFFFFFFFFFFFFull;
          bad_score |= mag > 0x7FF0000000000000ull || (ks != mag && mag != 0);
          key = (ks == 0x8000000000000000ull) ? 0ull : ks;  // -0 orders like +0
        }
      }
      // argmin of the 64-bit keys, ties to the lower server: minimum of the high
      // words, then of the low words among those lanes, then the lowest lane
      const unsigned khi = static_cast<unsigned>(key >> 32), klo = static_cast<unsigned>(key);
      const unsigned mhi = __reduce_min_sync(0xffffffffu, khi);
      const unsigned mlo = __reduce_min_sync(0xffffffffu, khi == mhi ? klo : 0xffffffffu);
      const unsigned win = __ballot_sync(0xffffffffu, khi == mhi && klo == mlo);
      int m = __ffs(win) - 1;
      if (mhi == 0xffffffffu && mlo == 0xffffffffu) m = 64;  // no feasible server
      if (m == 64) {
        if (t == 0) waiting[nw] = j;
        ++nw;
      } else if (t == m) {
        xs[m * 64 + j] = 1;
        eta[m * 64 + g] += 1;
        b = bn;
        a1 = a1n;
      }
      __syncwarp();
    }
    // waiting list: the server with the largest C_m - b_m (ties: lower m)
    for (int w = 0; w < nw; ++w) {
      const int j = waiting[w];
      const double room = srv ? __dsub_rn(cap, b) : -INFINITY;
      double br = room;
      int bm = srv ? t : 64;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const double orr = __shfl_xor_sync(0xffffffffu, br, o);
        const int om_ = __shfl_xor_sync(0xffffffffu, bm, o);
        if (orr > br || (orr == br && om_ < bm)) {
          br = orr;
          bm = om_;
        }
      }
      if (t == bm) {
        xs[bm * 64 + j] = 1;
        b = __dadd_rn(b, pls[j]);
        a1 = __dmul_rn(pp.lambda1, div_rn_markstein(b, cap, rcap));
        if (b > cap) overflow = 1;
      }
      __syncwarp();
    }
    uint8_t* x = placement + (size_t)l * M * E;
    for (int i = t; i < M * E; i += 32) x[i] = xs[(i / E) * 64 + (i % E)];
    __syncwarp();
  }
  if (srv) used[t] = b;
  overflow = __any_sync(0xffffffffu, overflow != 0);
  if (__any_sync(0xffffffffu, bad_score) && t == 0)
    report(&g_err_sim, ORDERMOE_DEV_BAD_VALUE, 0);
  return overflow;
}

// Eq. 29's memory over all layers against the servers' total (the capacity
// status of the first range), summed in order by one thread.
__device__ int demand_exceeds(const double* __restrict__ p, int n, const double* __restrict__ C,
                              int M) {
  double need = 0.0, have = 0.0;
  for (int i = 0; i < n; ++i) need = __dadd_rn(need, p[i]);
  for (int m = 0; m < M; ++m) have = __dadd_rn(have, C[m]);
  return need > have ? 1 : 0;
}

// Status of a placed range: the first range sets it, a later one only raises
// the capacity error.
__device__ void place_status(int first, int overflow, int32_t* __restrict__ status) {
  if (first || overflow) *status = overflow ? ORDERMOE_ERR_CAPACITY : ORDERMOE_OK;
}

__global__ void __launch_bounds__(64) place_kernel(
    const int32_t* __restrict__ group, const int32_t* __restrict__ porder, int L, int E, int M,
    int l0, int l1, int first, PlaceParams pp, const double* __restrict__ p,
    const double* __restrict__ C, uint8_t* __restrict__ placement, double* __restrict__ used,
    int32_t* __restrict__ status) {
  __shared__ PlaceSmem sm;
  __shared__ int s_over;
  int over = 0;
  if (threadIdx.x < 32)
    over = place_layers(sm, group, porder, L, E, M, l0, l1, first, pp, p, C, placement, used);
  else if (threadIdx.x == 32 && first)  // beside the placement, on the second warp
    s_over = demand_exceeds(p, L * E, C, M);
  __syncthreads();
  if (threadIdx.x == 0) place_status(first, over | (first ? s_over : 0), status);
}

// Grouping and placement of layers l0 .. l1 - 1 in one block: the grouping
// runs kGroupSlices layers at a time, 64 threads a layer; then warp 0 places
// the layers in order while the second warp sums the capacity check (one
// block, so the pipelined plan's side stream holds one SM).
constexpr int kGroupSlices = 4;
constexpr size_t kGroupPlaceSmem = kGroupSlices * sizeof(GroupSmem) + sizeof(PlaceSmem);

__global__ void __launch_bounds__(64 * kGroupSlices) group_place_kernel(
    const float* __restrict__ sim, const int32_t* __restrict__ counts, int L, int E, int M, int l0,
    int l1, int first, PlaceParams pp, const double* __restrict__ p, const double* __restrict__ C,
    int32_t* __restrict__ group, int32_t* __restrict__ n_groups, float* __restrict__ theta_out,
    double* __restrict__ importance, int32_t* __restrict__ porder, uint8_t* __restrict__ placement,
    double* __restrict__ used, int32_t* __restrict__ status) {
  extern __shared__ __align__(16) unsigned char s_gp[];
  GroupSmem* gs = reinterpret_cast<GroupSmem*>(s_gp);
  PlaceSmem& ps = *reinterpret_cast<PlaceSmem*>(s_gp + kGroupSlices * sizeof(GroupSmem));
  const int slice = threadIdx.x / 64;
  for (int lb = l0; lb < l1; lb += kGroupSlices) {
    const int l = lb + slice;
    group_layer(gs[slice], l < l1, threadIdx.x % 64, l, sim, counts, L, E, pp, p, group, n_groups,
                theta_out, importance, porder);
    __syncthreads();  // the slices' scratch is reused by the next round
  }
  // group and porder written above are visible to the block after the barrier
  __shared__ int s_over;
  int over = 0;
  if (threadIdx.x < 32)
    over = place_layers(ps, group, porder, L, E, M, l0, l1, first, pp, p, C, placement, used);
  else if (threadIdx.x == 32 && first)
    s_over = demand_exceeds(p, L * E, C, M);
  __syncthreads();
  if (threadIdx.x == 0) place_status(first, over | (first ? s_over : 0), status);
}

}  // namespace om

using namespace om;

namespace om {
bool sim_tc_supported(int L, int E);
int sim_tc_nsplit(int L, int E, int64_t N);
int sim_tc_max_splits();
int sim_tc_launch(const uint16_t* X, int N, const uint16_t* W, int L, int E, int d, int kf,
                  float* H, uint16_t* hi, uint16_t* lo, int ldT, int32_t* counts, float* gpart,
                  int nsplit, bool reserve_sm, cudaStream_t stream);
}  // namespace om

// Workspace: H [N][L E] fp32 | the hi/lo bf16 planes of H^T [L E][ldT] (tensor-core
// path) | partial Grams [L][parts][64][64] fp32 | G [L][64][64] fp64.
static int64_t sim_ldT(int64_t N) { return (N + 7) / 8 * 8; }

// Partial Grams per layer the workspace holds: one per 1024-token chunk on
// the CUDA-core path, one per token split (at most sim_tc_max_splits, and at
// most one per 64-token step) on the tensor-core path.
static int64_t sim_parts(int L, int E, int64_t N) {
  if (!sim_tc_supported(L, E)) return (N + kSimChunk - 1) / kSimChunk;
  const int64_t kb = (N + 63) / 64;
  return kb < sim_tc_max_splits() ? kb : sim_tc_max_splits();
}

// Workspace of the similarity: H [N][L E] fp32 (with_H; the CUDA-core path
// and the logits-keeping call need it), the hi/lo planes (tensor-core path),
// the partial Grams and G.
static size_t sim_ws_bytes(int L, int E, int64_t N, bool with_H) {
  if (L <= 0 || E <= 0 || E > ORDERMOE_MAX_EXPERTS || N <= 0) return 0;
  auto up = [](size_t v) { return (v + 255) & ~size_t(255); };
  const size_t h = with_H ? up((size_t)N * L * E * sizeof(float)) : 0;
  const size_t planes = sim_tc_supported(L, E) ? 2 * up((size_t)L * E * sim_ldT(N) * 2) : 0;
  const size_t g = (size_t)L * sim_parts(L, E, N) * 64 * 64 * sizeof(float);
  const size_t gd = (size_t)L * 64 * 64 * sizeof(double);
  return h + planes + up(g) + up(gd);
}

extern "C" size_t ordermoe_similarity_workspace_bytes(int L, int E, int64_t N) {
  return sim_ws_bytes(L, E, N, true);
}

// The similarity arguments a call needs (Eqs. 3-5), checked.
static int similarity_check(const uint16_t* W_r, const uint16_t* X_cal, int L, int E, int d,
                            int64_t N, int k_freq, const float* sim, const int32_t* counts,
                            const void* workspace, size_t workspace_bytes, size_t need_bytes) {
  if (L <= 0 || E <= 0 || E > ORDERMOE_MAX_EXPERTS || k_freq <= 0 || k_freq > E)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "similarity: need L >= 1, 1 <= k_freq <= E <= 64");
  if (d <= 0 || d % 64 != 0)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "similarity: d must be a positive multiple of 64");
  if (N <= 0 || N > 65535LL * kSimChunk || (int64_t)L * E > INT32_MAX || L > 65535)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "similarity: need 1 <= N <= 65535 * 1024");
  if (!W_r || !X_cal || !sim || !counts || !workspace)
    return fail(ORDERMOE_ERR_INVALID_ARG, "similarity: null pointer");
  if (!aligned16(W_r) || !aligned16(X_cal) || (reinterpret_cast<uintptr_t>(workspace) & 255u))
    return fail(ORDERMOE_ERR_INVALID_ARG, "similarity: W_r/X_cal 16-byte and workspace 256-byte aligned");
  if (workspace_bytes < need_bytes)
    return fail(ORDERMOE_ERR_INVALID_ARG, "similarity: workspace too small");
  return ORDERMOE_OK;
}

// Where the similarity's scratch lives in its workspace.
struct SimLayout {
  float* H;
  uint16_t* hi;
  uint16_t* lo;
  float* gpart;
  double* G;
  int64_t ldT;
  int nchunks;
  bool tc;
};

static SimLayout similarity_layout(void* workspace, int L, int E, int64_t N, bool with_H) {
  auto up = [](size_t v) { return (v + 255) & ~size_t(255); };
  SimLayout w;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  w.H = with_H ? reinterpret_cast<float*>(ws) : nullptr;
  w.tc = sim_tc_supported(L, E);
  w.nchunks = static_cast<int>((N + kSimChunk - 1) / kSimChunk);
  w.ldT = sim_ldT(N);
  const size_t plane = up((size_t)L * E * w.ldT * 2);
  w.hi = reinterpret_cast<uint16_t*>(ws + (with_H ? up((size_t)N * L * E * sizeof(float)) : 0));
  w.lo = reinterpret_cast<uint16_t*>(reinterpret_cast<uint8_t*>(w.hi) + plane);
  w.gpart = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(w.hi) + (w.tc ? 2 * plane : 0));
  w.G = reinterpret_cast<double*>(reinterpret_cast<uint8_t*>(w.gpart) +
                                  up((size_t)L * sim_parts(L, E, N) * 64 * 64 * sizeof(float)));
  return w;
}

// keep_logits: leave the fp32 calibration logits H in the workspace (the
// input of ordermoe_transitions); the tensor-core path can skip writing them.
static int similarity_impl(const uint16_t* W_r, const uint16_t* X_cal, int L, int E, int d,
                           int64_t N, int k_freq, float* sim, int32_t* counts, void* workspace,
                           size_t workspace_bytes, bool keep_logits, cudaStream_t stream) {
  int rc0 = similarity_check(W_r, X_cal, L, E, d, N, k_freq, sim, counts, workspace, workspace_bytes,
                             ordermoe_similarity_workspace_bytes(L, E, N));
  if (rc0) return rc0;
  const SimLayout w = similarity_layout(workspace, L, E, N, true);
  float* H = w.H;
  uint16_t* hi = w.hi;
  uint16_t* lo = w.lo;
  float* gpart = w.gpart;
  double* G = w.G;
  const bool tc = w.tc;
  const int64_t ldT = w.ldT;
  const int nchunks = w.nchunks;
  OM_CUDA(cudaMemsetAsync(counts, 0, sizeof(int32_t) * L * E, stream));
  if (tc) {
    // tensor-core path: logits with fused counts and hi/lo planes, then the Gram
    const int nsplit = sim_tc_nsplit(L, E, N);
    int rc = sim_tc_launch(X_cal, static_cast<int>(N), W_r, L, E, d, k_freq,
                           keep_logits ? H : nullptr, hi, lo, static_cast<int>(ldT), counts, gpart,
                           nsplit, false, stream);
    if (rc) return rc;
    gram_reduce_kernel<<<dim3(L, 16), 256, 0, stream>>>(gpart, nsplit, G);
    OM_LAUNCHED("gram_reduce_kernel");
    sim_finish_kernel<<<dim3(L, 16), 256, 0, stream>>>(G, E, sim);
    OM_LAUNCHED("sim_finish_kernel");
    return ORDERMOE_OK;
  }
  int rc = logits_gemm_launch(X_cal, static_cast<int>(N), W_r, L * E, d, H, stream);
  if (rc) return rc;
  int64_t cblocks = (N + 255) / 256;
  const int64_t ccap = (num_sms() * 8 + L - 1) / L;
  if (cblocks > ccap) cblocks = ccap;
  const dim3 cgrid(L, static_cast<unsigned>(cblocks));
  if (E <= 8) counts_kernel<8><<<cgrid, 256, 0, stream>>>(H, N, L, E, k_freq, counts);
  else if (E <= 16) counts_kernel<16><<<cgrid, 256, 0, stream>>>(H, N, L, E, k_freq, counts);
  else if (E <= 32) counts_kernel<32><<<cgrid, 256, 0, stream>>>(H, N, L, E, k_freq, counts);
  else counts_kernel<64><<<cgrid, 256, 0, stream>>>(H, N, L, E, k_freq, counts);
  OM_LAUNCHED("counts_kernel");
  gram_kernel<<<dim3(L, nchunks), 256, 0, stream>>>(H, N, L, E, gpart);
  OM_LAUNCHED("gram_kernel");
  gram_reduce_kernel<<<dim3(L, 16), 256, 0, stream>>>(gpart, nchunks, G);
  OM_LAUNCHED("gram_reduce_kernel");
  sim_finish_kernel<<<dim3(L, 16), 256, 0, stream>>>(G, E, sim);
  OM_LAUNCHED("sim_finish_kernel");
  return ORDERMOE_OK;
}

extern "C" int ordermoe_similarity(const uint16_t* W_r, const uint16_t* X_cal, int L, int E, int d,
                                   int64_t N, int k_freq, float* sim, int32_t* counts,
                                   void* workspace, size_t workspace_bytes,
                                   ordermoe_stream_t stream) {
  OM_TRACE();
  return similarity_impl(W_r, X_cal, L, E, d, N, k_freq, sim, counts, workspace, workspace_bytes,
                         true, stream);
}

extern "C" int ordermoe_similarity_no_logits(const uint16_t* W_r, const uint16_t* X_cal, int L,
                                             int E, int d, int64_t N, int k_freq, float* sim,
                                             int32_t* counts, void* workspace,
                                             size_t workspace_bytes, ordermoe_stream_t stream) {
  OM_TRACE();
  return similarity_impl(W_r, X_cal, L, E, d, N, k_freq, sim, counts, workspace, workspace_bytes,
                         false, stream);
}

extern "C" int ordermoe_expert_counts(const float* logits, int64_t N, int E, int k_freq,
                                      int32_t* counts, ordermoe_stream_t stream) {
  OM_TRACE();
  if (E <= 0 || E > ORDERMOE_MAX_EXPERTS || k_freq <= 0 || k_freq > E || N < 0)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "expert_counts: need 1 <= k_freq <= E <= 64");
  if (!counts || (N > 0 && !logits)) return fail(ORDERMOE_ERR_INVALID_ARG, "expert_counts: null pointer");
  OM_CUDA(cudaMemsetAsync(counts, 0, sizeof(int32_t) * E, stream));
  if (N == 0) return ORDERMOE_OK;
  int64_t blocks = (N + 255) / 256;
  if (blocks > num_sms() * 4) blocks = num_sms() * 4;
  counts_from_logits_kernel<<<static_cast<int>(blocks), 256, 0, stream>>>(logits, N, E, k_freq, counts);
  OM_LAUNCHED("counts_from_logits_kernel");
  return ORDERMOE_OK;
}

namespace om {

constexpr int kRepThreads = 512;
constexpr int kRepMaxCand = 16384;
constexpr int kRepMaxLayers = 1024;

// Redundant deployment for one server (blockIdx.x = m), Eqs. 32-35. The
// candidates (l, j) get the key (benefit bits, then candidate id), are sorted
// by benefit desc and id asc (bitonic sort in shared memory), and are deployed
// in that order while the group is uncovered and the replica fits. Benefits
// are positive fp64 values, so their bit patterns order like the values;
// non-positive and NaN benefits get key 0 and are never taken. A server's
// state (b_m and its covered groups) changes only when it takes a candidate,
// so one warp tests 32 sorted candidates at a time against the current state
// and takes the first that passes: every candidate it passes over failed
// under the same state it would have met one at a time.
__global__ void __launch_bounds__(kRepThreads) replicate_kernel(
    const int32_t* __restrict__ group, const double* __restrict__ importance,
    const double* __restrict__ p, const double* __restrict__ C, const double* __restrict__ pi,
    int L, int E, int M, int Np, uint8_t* __restrict__ placement, double* __restrict__ used,
    int32_t* __restrict__ replicas) {
  extern __shared__ __align__(16) unsigned char s_rep[];
  unsigned long long* key = reinterpret_cast<unsigned long long*>(s_rep);
  unsigned long long* cov = key + Np;  // [L]: bit g = group g covered (Eq. 32)
  uint32_t* cid = reinterpret_cast<uint32_t*>(cov + L);
  const int m = blockIdx.x;
  const int t = threadIdx.x;
  const int N = L * E;
  for (int l = t; l < L; l += blockDim.x) {
    unsigned long long bits = 0;
    for (int j = 0; j < E; ++j) {
      const int g = group[(size_t)l * E + j];
      if (placement[((size_t)l * M + m) * E + j] && g >= 0 && g < E) bits |= 1ull << g;
    }
    cov[l] = bits;
  }
  const double pim = pi[m];
  for (int i = t; i < Np; i += blockDim.x) {
    unsigned long long k = 0;
    if (i < N) {
      const int g = group[i];
      const double pj = p[i];
      if (g < 0 || g >= E) {
        if (m == 0) report(&g_err_sim, ORDERMOE_DEV_BAD_INDEX, i);
      } else if (!(pj > 0.0)) {
        if (m == 0) report(&g_err_sim, ORDERMOE_DEV_BAD_VALUE, i);
      } else {
        const double ben = __ddiv_rn(__dmul_rn(pim, importance[i]), pj);  // Eq. 33, y = 0
        if (ben > 0.0) k = static_cast<unsigned long long>(__double_as_longlong(ben));
      }
    }
    key[i] = k;
    cid[i] = i < N ? static_cast<uint32_t>(i) : 0xFFFFFFFFu;
  }
  __syncthreads();
  // bitonic sort into (key desc, cid asc)
  for (int size = 2; size <= Np; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = t; i < Np; i += blockDim.x) {
        const int o = i ^ stride;
        if (o > i) {
          const unsigned long long ki = key[i], ko = key[o];
          const uint32_t ci = cid[i], co = cid[o];
          const bool o_first = ko > ki || (ko == ki && co < ci);
          const bool i_first = ki > ko || (ki == ko && ci < co);
          if ((i & size) == 0 ? o_first : i_first) {
            key[i] = ko; key[o] = ki;
            cid[i] = co; cid[o] = ci;
          }
        }
      }
      __syncthreads();
    }
  }
  // the candidates (key != 0) are a prefix of the sorted order; each sorted
  // slot is repacked in place as (l, g, j) and the bits of p_{l,j}
  __shared__ int n_cand;
  if (t == 0) n_cand = 0;
  __syncthreads();
  int mine = 0;
  for (int s = t; s < N; s += blockDim.x) {
    if (key[s] == 0) continue;
    ++mine;
    const int i = static_cast<int>(cid[s]);
    const int l = i / E, j = i - l * E;
    cid[s] = (static_cast<uint32_t>(l) << 12) | (static_cast<uint32_t>(group[i]) << 6) |
             static_cast<uint32_t>(j);
    key[s] = static_cast<unsigned long long>(__double_as_longlong(p[i]));
  }
  if (mine) atomicAdd(&n_cand, mine);
  __syncthreads();
  if (t < 32) {
    const unsigned full = 0xffffffffu;
    const int nc = n_cand;
    double b = used[m];
    const double cap = C[m];
    int count = 0;
    for (int base = 0; base < nc;) {
      const int s = base + t;
      uint32_t rec = 0;
      double pj = 0.0;
      bool take = false;
      if (s < nc) {
        rec = cid[s];
        pj = __longlong_as_double(static_cast<long long>(key[s]));
        const int l = static_cast<int>(rec >> 12), g = static_cast<int>((rec >> 6) & 63u);
        take = !((cov[l] >> g) & 1ull) &&        // B = 0 once the group is local
               __dadd_rn(b, pj) <= cap;          // Eq. 35
      }
      const unsigned bal = __ballot_sync(full, take);
      if (bal == 0) {
        base += 32;
        continue;
      }
      const int w = __ffs(bal) - 1;
      if (t == w) {
        const int l = static_cast<int>(rec >> 12), g = static_cast<int>((rec >> 6) & 63u);
        placement[((size_t)l * M + m) * E + static_cast<int>(rec & 63u)] = 1;
        cov[l] |= 1ull << g;
      }
      b = __dadd_rn(b, __shfl_sync(full, pj, w));
      ++count;
      base += w + 1;
      __syncwarp();
    }
    if (t == 0) {
      used[m] = b;
      replicas[m] = count;
    }
  }
}

// Eq. 32 for one layer (blockIdx.x = l): thread m ORs its server's groups.
__global__ void __launch_bounds__(32) coverage_kernel(const int32_t* __restrict__ group,
                                                      const uint8_t* __restrict__ placement, int L,
                                                      int E, int M, uint8_t* __restrict__ cover,
                                                      int32_t* __restrict__ covered) {
  const int l = blockIdx.x;
  const int m = threadIdx.x;
  // the layer's groups, checked once (-1: out of range, reported)
  __shared__ int gsh[64];
  for (int j = m; j < E; j += 32) {
    int g = group[(size_t)l * E + j];
    if (g < 0 || g >= E) {
      report(&g_err_sim, ORDERMOE_DEV_BAD_INDEX, l * E + j);
      g = -1;
    }
    gsh[j] = g;
  }
  __syncwarp();
  // server m's row of the layer's placement: 16-byte loads where it allows,
  // all issued before they are used
  unsigned long long bits = 0;
  if (m < M) {
    const uint8_t* row = placement + ((size_t)l * M + m) * E;
    if ((E & 15) == 0 && (reinterpret_cast<uintptr_t>(row) & 15u) == 0) {
      uint4 v[4];
#pragma unroll
      for (int c = 0; c < 4; ++c)
        if (c < E / 16) v[c] = reinterpret_cast<const uint4*>(row)[c];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        if (c >= E / 16) break;
        const uint32_t w[4] = {v[c].x, v[c].y, v[c].z, v[c].w};
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const int g = gsh[c * 16 + q];
          if (((w[q >> 2] >> (8 * (q & 3))) & 0xFFu) != 0u && g >= 0) bits |= 1ull << g;
        }
      }
    } else {
#pragma unroll 16
      for (int j = 0; j < E; ++j) {
        const int g = gsh[j];
        if (row[j] && g >= 0) bits |= 1ull << g;
      }
    }
  }
  if (m < M && cover != nullptr)
    for (int g = 0; g < E; ++g) cover[((size_t)l * M + m) * E + g] = (bits >> g) & 1ull;
  int n = __popcll(bits);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
  if (m == 0 && covered != nullptr) covered[l] = n;
}

}  // namespace om

extern "C" size_t ordermoe_place_workspace_bytes(int L, int E) {
  if (L <= 0 || E <= 0 || E > ORDERMOE_MAX_EXPERTS) return 0;
  return ((size_t)L * E * sizeof(int32_t) + 255) & ~size_t(255);
}

extern "C" int ordermoe_place(const float* sim, const int32_t* counts, int L, int E, int M,
                              double theta_min, double theta_max, double theta_single,
                              double alpha_f, double alpha_r, double lambda1, double lambda2,
                              const double* p, const double* C, int32_t* group, int32_t* n_groups,
                              float* theta, double* importance, uint8_t* placement, double* used,
                              int32_t* status, void* workspace, size_t workspace_bytes,
                              ordermoe_stream_t stream) {
  OM_TRACE();
  if (L <= 0 || E <= 0 || E > ORDERMOE_MAX_EXPERTS || M <= 0 || M > ORDERMOE_MAX_SERVERS)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "place: need L >= 1, 1 <= E <= 64, 1 <= M <= 32");
  if (!sim || !counts || !p || !C || !group || !n_groups || !theta || !placement || !used || !status)
    return fail(ORDERMOE_ERR_INVALID_ARG, "place: null pointer");
  if (!workspace || workspace_bytes < ordermoe_place_workspace_bytes(L, E))
    return fail(ORDERMOE_ERR_INVALID_ARG, "place: workspace missing or too small");
  int32_t* porder_scratch = static_cast<int32_t*>(workspace);
  PlaceParams pp{theta_min, theta_max, theta_single, alpha_f, alpha_r, lambda1, lambda2};
  group_kernel<<<L, 64, 0, stream>>>(sim, counts, L, E, 0, pp, p, group, n_groups, theta, importance,
                                     porder_scratch);
  OM_LAUNCHED("group_kernel");
  place_kernel<<<1, 64, 0, stream>>>(group, porder_scratch, L, E, M, 0, L, 1, pp, p, C, placement,
                                     used, status);
  OM_LAUNCHED("place_kernel");
  return ORDERMOE_OK;
}

static int transitions_launch(const char* who, const float* logits, int64_t N, int L, int E,
                              int k_freq, int64_t sn, int64_t sl, int32_t* counts, float* P,
                              cudaStream_t stream) {
  if (L < 2 || E <= 0 || E > ORDERMOE_MAX_EXPERTS || k_freq <= 0 || k_freq > E || N < 0)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "%s: need L >= 2, 1 <= k_freq <= E <= 64", who);
  if (!counts || !P || (N > 0 && !logits)) return fail(ORDERMOE_ERR_INVALID_ARG, "%s: null pointer", who);
  OM_CUDA(cudaMemsetAsync(counts, 0, sizeof(int32_t) * (size_t)(L - 1) * E * E, stream));
  if (N > 0) {
    int64_t blocks = (N + 255) / 256;
    const int64_t cap = (num_sms() * 4 + L - 2) / (L - 1);
    if (blocks > cap) blocks = cap;
    const dim3 grid(static_cast<unsigned>(blocks), L - 1);
    if (E <= 8) transitions_kernel<8><<<grid, 256, 0, stream>>>(logits, N, L, E, k_freq, sn, sl, counts);
    else if (E <= 16) transitions_kernel<16><<<grid, 256, 0, stream>>>(logits, N, L, E, k_freq, sn, sl, counts);
    else if (E <= 32) transitions_kernel<32><<<grid, 256, 0, stream>>>(logits, N, L, E, k_freq, sn, sl, counts);
    else transitions_kernel<64><<<grid, 256, 0, stream>>>(logits, N, L, E, k_freq, sn, sl, counts);
    OM_LAUNCHED("transitions_kernel");
  }
  const int rows = (L - 1) * E;
  transitions_finish_kernel<<<(rows + 127) / 128, 128, 0, stream>>>(counts, rows, E, P);
  OM_LAUNCHED("transitions_finish_kernel");
  return ORDERMOE_OK;
}

extern "C" int ordermoe_transitions(const float* logits, int64_t N, int L, int E, int k_freq,
                                    int32_t* counts, float* P, ordermoe_stream_t stream) {
  OM_TRACE();
  return transitions_launch("transitions", logits, N, L, E, k_freq, (int64_t)L * E, E, counts, P,
                            stream);
}

extern "C" int ordermoe_transitions_strided(const float* logits, int64_t N, int L, int E,
                                            int k_freq, int64_t token_stride, int64_t layer_stride,
                                            int32_t* counts, float* P, ordermoe_stream_t stream) {
  OM_TRACE();
  if (token_stride < E || layer_stride < E)
    return fail(ORDERMOE_ERR_INVALID_ARG, "transitions_strided: strides must be >= E");
  return transitions_launch("transitions_strided", logits, N, L, E, k_freq, token_stride,
                            layer_stride, counts, P, stream);
}

extern "C" int ordermoe_replicate(const int32_t* group, const double* importance, const double* p,
                                  const double* C, const double* pi, int L, int E, int M,
                                  uint8_t* placement, double* used, int32_t* replicas,
                                  ordermoe_stream_t stream) {
  OM_TRACE();
  if (L <= 0 || L > kRepMaxLayers || E <= 0 || E > ORDERMOE_MAX_EXPERTS || M <= 0 ||
      M > ORDERMOE_MAX_SERVERS || (long long)L * E > kRepMaxCand)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE,
                "replicate: need 1 <= L <= 1024, 1 <= E <= 64, L * E <= 16384, 1 <= M <= 32");
  if (!group || !importance || !p || !C || !pi || !placement || !used || !replicas)
    return fail(ORDERMOE_ERR_INVALID_ARG, "replicate: null pointer");
  int Np = 1;
  while (Np < L * E) Np <<= 1;
  const size_t smem = (size_t)Np * (sizeof(unsigned long long) + sizeof(uint32_t)) +
                      (size_t)L * sizeof(unsigned long long);
  // once per device, for the largest sort (no attribute call per launch, so
  // the call can be captured into a CUDA graph)
  static PerDevice attr;
  const cudaError_t ae = static_cast<cudaError_t>(per_device(attr, [] {
    const size_t most = (size_t)kRepMaxCand * (sizeof(unsigned long long) + sizeof(uint32_t)) +
                        (size_t)kRepMaxLayers * sizeof(unsigned long long);
    return static_cast<int>(cudaFuncSetAttribute(
        replicate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)most));
  }));
  if (ae != cudaSuccess) return cuda_fail(ae, "cudaFuncSetAttribute(replicate_kernel)");
  replicate_kernel<<<M, kRepThreads, smem, stream>>>(group, importance, p, C, pi, L, E, M, Np,
                                                     placement, used, replicas);
  OM_LAUNCHED("replicate_kernel");
  return ORDERMOE_OK;
}

extern "C" int ordermoe_coverage(const int32_t* group, const uint8_t* placement, int L, int E,
                                 int M, uint8_t* cover, int32_t* covered,
                                 ordermoe_stream_t stream) {
  OM_TRACE();
  if (L <= 0 || E <= 0 || E > ORDERMOE_MAX_EXPERTS || M <= 0 || M > ORDERMOE_MAX_SERVERS)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "coverage: need L >= 1, 1 <= E <= 64, 1 <= M <= 32");
  if (!group || !placement) return fail(ORDERMOE_ERR_INVALID_ARG, "coverage: null pointer");
  coverage_kernel<<<L, 32, 0, stream>>>(group, placement, L, E, M, cover, covered);
  OM_LAUNCHED("coverage_kernel");
  return ORDERMOE_OK;
}

extern "C" int ordermoe_selftest_div_rn(const double* a, const double* b, double* out, int64_t n,
                                        ordermoe_stream_t stream) {
  OM_TRACE();
  if (n < 0) return fail(ORDERMOE_ERR_INVALID_ARG, "selftest_div_rn: n < 0");
  if (n == 0) return ORDERMOE_OK;
  if (!a || !b || !out) return fail(ORDERMOE_ERR_INVALID_ARG, "selftest_div_rn: null pointer");
  int64_t blocks = (n + 255) / 256;
  if (blocks > num_sms() * 8) blocks = num_sms() * 8;
  div_selftest_kernel<<<static_cast<int>(blocks), 256, 0, stream>>>(a, b, out, n);
  OM_LAUNCHED("div_selftest_kernel");
  return ORDERMOE_OK;
}

// ----------------------------------------------------------------------------
// The whole offline plan in one call (Alg. 1): similarity (Eqs. 3-5), grouping
// (Eqs. 6, 24-28), mandatory placement (Eqs. 29-31), redundant deployment
// (Eqs. 32-35) and coverage (Eq. 32). On the tensor-core path the layers go in
// blocks of 512 logit columns (the last block in two halves when there are
// several): the caller's stream runs a block's logits GEMM,
// Gram and similarities, and a side stream, behind an event, runs that
// block's grouping and placement while the next block's GEMM runs. The
// placement carries b_m from block to block in `used`; its layers stay in
// order because the side stream runs the blocks in order. The results are
// those of ordermoe_similarity_no_logits, ordermoe_place, ordermoe_replicate
// and ordermoe_coverage called one after the other.
namespace om {

int sim_tc_part_layers(int E);

// One side stream and its events per device, shared by every call: a call
// holds `mu` while it enqueues, so calls from several host threads cannot
// interleave their event records (a stream wait takes the event as it was
// when the wait was enqueued).
struct PlanSync {
  std::mutex mu;
  cudaStream_t side;
  cudaEvent_t ev[4];
};
static PlanSync g_plan_sync[64];
static PerDevice g_plan_sync_once;

static int plan_sync(PlanSync** out) {
  int dev = 0;
  OM_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 64) return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "plan: device index above 63");
  const int e = per_device(g_plan_sync_once, [dev] {
    PlanSync& ps = g_plan_sync[dev];
    cudaError_t err = cudaFuncSetAttribute(group_place_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           static_cast<int>(kGroupPlaceSmem));
    if (err == cudaSuccess) err = cudaStreamCreateWithFlags(&ps.side, cudaStreamNonBlocking);
    for (int i = 0; i < 4 && err == cudaSuccess; ++i)
      err = cudaEventCreateWithFlags(&ps.ev[i], cudaEventDisableTiming);
    return static_cast<int>(err);
  });
  if (e != cudaSuccess) return cuda_fail(static_cast<cudaError_t>(e), "plan: side stream and events");
  *out = &g_plan_sync[dev];
  return ORDERMOE_OK;
}

static int launched(const char* what) {
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? ORDERMOE_OK : cuda_fail(e, what);
}

}  // namespace om

// The similarity part of the plan's workspace: without H on the tensor-core
// path (the plan keeps no logits), the whole similarity workspace otherwise.
static size_t plan_sim_bytes(int L, int E, int64_t N) {
  return sim_ws_bytes(L, E, N, !sim_tc_supported(L, E));
}

extern "C" size_t ordermoe_plan_workspace_bytes(int L, int E, int64_t N) {
  const size_t a = plan_sim_bytes(L, E, N);  // a multiple of 256
  const size_t b = ordermoe_place_workspace_bytes(L, E);
  return (a == 0 || b == 0) ? 0 : a + b;
}

extern "C" int ordermoe_plan(const uint16_t* W_r, const uint16_t* X_cal, int L, int E, int d,
                             int64_t N, int k_freq, int M, double theta_min, double theta_max,
                             double theta_single, double alpha_f, double alpha_r, double lambda1,
                             double lambda2, const double* p, const double* C, const double* pi,
                             float* sim, int32_t* counts, int32_t* group, int32_t* n_groups,
                             float* theta, double* importance, uint8_t* placement, double* used,
                             int32_t* status, int32_t* replicas, uint8_t* cover, int32_t* covered,
                             void* workspace, size_t workspace_bytes, ordermoe_stream_t stream) {
  OM_TRACE();
  const size_t sim_ws = plan_sim_bytes(L, E, N);
  int rc = similarity_check(W_r, X_cal, L, E, d, N, k_freq, sim, counts, workspace, sim_ws, sim_ws);
  if (rc) return rc;
  if (M <= 0 || M > ORDERMOE_MAX_SERVERS || L > kRepMaxLayers || (long long)L * E > kRepMaxCand)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE,
                "plan: need 1 <= M <= 32, L <= 1024 and L * E <= 16384");
  if (!p || !C || !pi || !group || !n_groups || !theta || !importance || !placement || !used ||
      !status || !replicas)
    return fail(ORDERMOE_ERR_INVALID_ARG, "plan: null pointer");
  if (workspace_bytes < ordermoe_plan_workspace_bytes(L, E, N))
    return fail(ORDERMOE_ERR_INVALID_ARG, "plan: workspace too small");
  int32_t* porder = reinterpret_cast<int32_t*>(static_cast<uint8_t*>(workspace) + sim_ws);
  const size_t porder_bytes = workspace_bytes - sim_ws;
  cudaStream_t S = static_cast<cudaStream_t>(stream);
  const SimLayout w = similarity_layout(workspace, L, E, N, !sim_tc_supported(L, E));
  if (!w.tc) {  // the CUDA-core similarity needs every layer's logits at once
    rc = similarity_impl(W_r, X_cal, L, E, d, N, k_freq, sim, counts, workspace, sim_ws, false, S);
    if (!rc)
      rc = ordermoe_place(sim, counts, L, E, M, theta_min, theta_max, theta_single, alpha_f, alpha_r,
                          lambda1, lambda2, p, C, group, n_groups, theta, importance, placement,
                          used, status, porder, porder_bytes, stream);
  } else {
    PlanSync* ps = nullptr;
    if ((rc = plan_sync(&ps))) return rc;
    std::lock_guard<std::mutex> hold(ps->mu);
    OM_CUDA(cudaMemsetAsync(counts, 0, sizeof(int32_t) * L * E, S));
    OM_CUDA(cudaEventRecord(ps->ev[0], S));
    OM_CUDA(cudaStreamWaitEvent(ps->side, ps->ev[0], 0));
    const PlaceParams pp{theta_min, theta_max, theta_single, alpha_f, alpha_r, lambda1, lambda2};
    const int part = sim_tc_part_layers(E);
    const int nsplit = sim_tc_nsplit(L, E, N);
    // the last block's grouping and placement are not hidden behind a GEMM:
    // when there is more than one block, the last one goes in two halves
    const int nfull = (L + part - 1) / part;
    const int last0 = (nfull - 1) * part, last_n = L - last0;
    for (int l0 = 0, k = 0; l0 < L && !rc; ++k) {
      int lp = L - l0 < part ? L - l0 : part;
      if (nfull > 1 && l0 >= last0 && last_n >= 2) lp = l0 == last0 ? (last_n + 1) / 2 : L - l0;
      const size_t rows = (size_t)l0 * E;
      float* gpart = w.gpart + (size_t)l0 * nsplit * 4096;
      double* G = w.G + (size_t)l0 * 4096;
      rc = sim_tc_launch(X_cal, static_cast<int>(N), W_r + rows * d, lp, E, d, k_freq, nullptr,
                         w.hi + rows * w.ldT, w.lo + rows * w.ldT, static_cast<int>(w.ldT),
                         counts + rows, gpart, nsplit, true, S);
      if (rc) break;
      gram_reduce_kernel<<<dim3(lp, 16), 256, 0, S>>>(gpart, nsplit, G);
      if ((rc = launched("gram_reduce_kernel"))) break;
      sim_finish_kernel<<<dim3(lp, 16), 256, 0, S>>>(G, E, sim + rows * E);
      if ((rc = launched("sim_finish_kernel"))) break;
      cudaEvent_t ev = ps->ev[1 + (k & 1)];
      cudaError_t e = cudaEventRecord(ev, S);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(ps->side, ev, 0);
      if (e != cudaSuccess) {
        rc = cuda_fail(e, "plan: block event");
        break;
      }
      group_place_kernel<<<1, 64 * kGroupSlices, kGroupPlaceSmem, ps->side>>>(
          sim, counts, L, E, M, l0, l0 + lp, l0 == 0 ? 1 : 0, pp, p, C, group, n_groups, theta,
          importance, porder, placement, used, status);
      if ((rc = launched("group_place_kernel"))) break;
      l0 += lp;
    }
    // every exit after the fork joins the side stream back into the caller's
    cudaError_t e = cudaEventRecord(ps->ev[3], ps->side);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(S, ps->ev[3], 0);
    if (!rc && e != cudaSuccess) rc = cuda_fail(e, "plan: join");
  }
  if (!rc)
    rc = ordermoe_replicate(group, importance, p, C, pi, L, E, M, placement, used, replicas, stream);
  if (!rc) rc = ordermoe_coverage(group, placement, L, E, M, cover, covered, stream);
  return rc;
}
