// ReSS block selection on sm_103a: pooling, pooled attention map, drift scoring, initial
// top-c selection and the restoration rounds (Sec. 4.1-4.3 of the paper).  This file holds
// pooling, the F-space projection, the per-row selection kernels and the kept-block lists;
// the row-by-block products (pooled logits, q, round gains) run on the tensor cores in
// k_dot.cu and the pooled map with y~ in k_yagg.cu.
//
// Arithmetic is float32 with fixed-order reductions (deterministic, Appendix B.4).  The
// per-head Gram matrix M_h = W_O^h^T W_O^h (Eq. 8) enters through its Cholesky factor F_h
// (F_h^T F_h = M_h), so every quadratic form of the method is a squared norm in the
// 64-dimensional "F space":
//   z~_j = F_h V_j,  y~_i = F_h v_bar_i = sum_j P_ij z~_j            (Eq. 1)
//   q_ij = ||y~_i - z~_j||^2 = e_ij^T M_h e_ij                     (Eq. 9, never negative)
//   g~   = F_h g = sum_{j in D} P_ij (y~_i - z~_j) = -sum_{j not in D} P_ij (y~_i - z~_j)
//   G    = ||g~||^2,  d_ik^T M_h g = P_ik (y~_i - z~_k) . g~        (Eq. 12, 14, 15)
// The last identity for g~ holds because sum_{j in B} P_ij (y~_i - z~_j) = 0: the net drift
// of the drop set is minus that of the kept set, which is the smaller one at high sparsity.

#include <math.h>
#include <stddef.h>

#include "ress_internal.cuh"
#include "sm100_ptx.cuh"

namespace ress {

constexpr int kThreads = 256;
constexpr unsigned kFull = 0xffffffffu;

// ------------------------------------------------------------------------------------
// Eq. 8: M_h = W_O^h^T W_O^h in float64, then its Cholesky factor F_h = L^T.
// ------------------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_prepare_wo(const uint16_t* __restrict__ W,
                                                          int d_model, int H,
                                                          float* __restrict__ F) {
  __shared__ double M[64][65];
  __shared__ double Wc[16][64];
  __shared__ double piv_s;
  const int h = blockIdx.x, t = threadIdx.x;
  const int a = t >> 2;  // row of M owned by this thread
  double acc[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) acc[k] = 0.0;
  const int64_t ldw = (int64_t)H * kHeadDim;
  for (int r0 = 0; r0 < d_model; r0 += 16) {
    for (int f = t; f < 16 * 64; f += kThreads) {
      const int rr = f >> 6, c = f & 63;
      double v = 0.0;
      if (r0 + rr < d_model) {
        const uint16_t b = W[(int64_t)(r0 + rr) * ldw + h * kHeadDim + c];
        v = (double)__uint_as_float((uint32_t)b << 16);
      }
      Wc[rr][c] = v;
    }
    __syncthreads();
    for (int rr = 0; rr < 16; ++rr) {
      const double wa = Wc[rr][a];
#pragma unroll
      for (int k = 0; k < 16; ++k) acc[k] += wa * Wc[rr][(t & 3) + 4 * k];
    }
    __syncthreads();
  }
#pragma unroll
  for (int k = 0; k < 16; ++k) M[a][(t & 3) + 4 * k] = acc[k];
  __syncthreads();
  // pivot tolerance relative to the largest diagonal entry
  if (t == 0) {
    double mx = 0.0;
    for (int k = 0; k < 64; ++k) mx = fmax(mx, M[k][k]);
    piv_s = mx * 1e-13;
  }
  __syncthreads();
  const double tol = piv_s;
  for (int k = 0; k < 64; ++k) {
    if (t == 0) {
      const double d = M[k][k];
      M[k][k] = d > tol ? sqrt(d) : 0.0;
    }
    __syncthreads();
    const double p = M[k][k];
    for (int i = k + 1 + t; i < 64; i += kThreads) M[i][k] = p > 0.0 ? M[i][k] / p : 0.0;
    __syncthreads();
    const int n = 63 - k;
    for (int idx = t; idx < n * n; idx += kThreads) {
      const int i = k + 1 + idx / n, j = k + 1 + idx % n;
      if (j <= i) M[i][j] -= M[i][k] * M[j][k];
    }
    __syncthreads();
  }
  // F[a][b] = L[b][a] for b >= a (upper triangular)
  for (int f = t; f < 64 * 64; f += kThreads) {
    const int r = f >> 6, c = f & 63;
    F[(int64_t)h * 4096 + f] = c >= r ? (float)M[c][r] : 0.0f;
  }
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// ------------------------------------------------------------------------------------
// Sec. 3 step (1): block means of Q (over query blocks of qb tokens), K and V (over 64-token
// key blocks), each over the valid tokens of its block.  grid (nb, 3); one token is H*64
// bf16 = 8H 16-byte chunks (H <= 32).
// ------------------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_pool(const uint16_t* __restrict__ Q,
                                                    const uint16_t* __restrict__ K,
                                                    const uint16_t* __restrict__ V, int N,
                                                    int H, int nb, int qb, int nq,
                                                    float* __restrict__ qbar,
                                                    float* __restrict__ kbar,
                                                    float* __restrict__ vbar,
                                                    uint16_t* __restrict__ qsplit,
                                                    uint16_t* __restrict__ ksplit) {
  __shared__ float part[kThreads * 8];
  const int j = blockIdx.x, which = blockIdx.y;
  const int bs = which == 0 ? qb : kBlock;        // tokens per block
  const int nblocks = which == 0 ? nq : nb;
  if (j >= nblocks) return;
  const uint16_t* X = which == 0 ? Q : (which == 1 ? K : V);
  float* out = which == 0 ? qbar : (which == 1 ? kbar : vbar);
  uint16_t* terms = which == 0 ? qsplit : (which == 1 ? ksplit : nullptr);  // tensor-core operands
  const int64_t term_stride = (int64_t)H * nblocks * kHeadDim;
  const int C = 8 * H;
  const int tpp = kThreads / C;
  const int tok0 = j * bs;
  const int valid = min(bs, N - tok0);
  const int c = threadIdx.x % C, slot = threadIdx.x / C;
  float acc[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) acc[e] = 0.f;
  if (slot < tpp) {
    const uint4* base = reinterpret_cast<const uint4*>(X + (int64_t)tok0 * H * kHeadDim) + c;
#pragma unroll 4
    for (int tk = slot; tk < valid; tk += tpp) {
      const uint4 v = ld_stream(base + (int64_t)tk * C);
      acc[0] += bf16_lo(v.x); acc[1] += bf16_hi(v.x);
      acc[2] += bf16_lo(v.y); acc[3] += bf16_hi(v.y);
      acc[4] += bf16_lo(v.z); acc[5] += bf16_hi(v.z);
      acc[6] += bf16_lo(v.w); acc[7] += bf16_hi(v.w);
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) part[slot * C * 8 + c * 8 + e] = acc[e];
  }
  __syncthreads();
  const float inv = 1.0f / (float)valid;
  for (int f = threadIdx.x; f < C * 8; f += kThreads) {
    float s = 0.f;
    for (int sl = 0; sl < tpp; ++sl) s += part[sl * C * 8 + f];
    const int h = f >> 6, d = f & 63;
    const int64_t at = ((int64_t)h * nblocks + j) * kHeadDim + d;
    out[at] = s * inv;
    if (terms) {
      uint16_t hi, mid, lo;
      split3_bf16(s * inv, hi, mid, lo);
      terms[at] = hi;
      terms[at + term_stride] = mid;
      terms[at + 2 * term_stride] = lo;
    }
  }
}

// ------------------------------------------------------------------------------------
// z~_j = F_h V_j.  grid (ceil(nb/16), H); thread (channel a, blocks 4q..4q+3 of the 16).
// F_h and the 16 pooled values sit in shared memory with rows padded to 68 floats, so that
// the float4 reads of a warp (32 channels, one column group) hit every bank once per pass.
// ------------------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_zproj(const float* __restrict__ F,
                                                     const float* __restrict__ vbar, int nb,
                                                     float* __restrict__ ztil,
                                                     uint16_t* __restrict__ zsplit,
                                                     int64_t term_stride,
                                                     float* __restrict__ nz) {
  constexpr int kPad = 68;
  __shared__ __align__(16) float Fs[64][kPad];  // Fs[a][b] = F[a][b]
  __shared__ __align__(16) float Vs[16][kPad];
  __shared__ float npart[8][4];
  const int h = blockIdx.y, j0 = blockIdx.x * 16, t = threadIdx.x;
  const int warp = t >> 5, lane = t & 31;
  for (int f = t; f < 1024; f += kThreads) {  // float4 units
    const int r = f >> 4, c4 = (f & 15) * 4;
    *reinterpret_cast<float4*>(&Fs[r][c4]) =
        *reinterpret_cast<const float4*>(F + (int64_t)h * 4096 + r * 64 + c4);
  }
  for (int f = t; f < 256; f += kThreads) {
    const int r = f >> 4, c4 = (f & 15) * 4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (j0 + r < nb) v = *reinterpret_cast<const float4*>(vbar + ((int64_t)h * nb + j0 + r) * 64 + c4);
    *reinterpret_cast<float4*>(&Vs[r][c4]) = v;
  }
  __syncthreads();
  const int a = t & 63, q = t >> 6;  // q is uniform across a warp
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
  for (int b4 = 0; b4 < 64; b4 += 4) {
    const float4 f = *reinterpret_cast<const float4*>(&Fs[a][b4]);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float4 v = *reinterpret_cast<const float4*>(&Vs[4 * q + u][b4]);
      acc[u] = fmaf(f.x, v.x, acc[u]);
      acc[u] = fmaf(f.y, v.y, acc[u]);
      acc[u] = fmaf(f.z, v.z, acc[u]);
      acc[u] = fmaf(f.w, v.w, acc[u]);
    }
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int j = j0 + 4 * q + u;
    if (j < nb) {
      const int64_t at = ((int64_t)h * nb + j) * 64 + a;
      ztil[at] = acc[u];
      // the same vector as three bf16 terms: an operand of the tensor-core products
      uint16_t hi, mid, lo;
      split3_bf16(acc[u], hi, mid, lo);
      zsplit[at] = hi;
      zsplit[at + term_stride] = mid;
      zsplit[at + 2 * term_stride] = lo;
    }
    const float n2 = warp_sum(acc[u] * acc[u]);  // this warp's 32 channels
    if (lane == 0) npart[warp][u] = n2;
  }
  __syncthreads();
  if (t < 16) {  // ||z~_j||^2: the two warps of block group q, fixed order
    const int qq = t >> 2, u = t & 3, j = j0 + t;
    if (j < nb) nz[(int64_t)h * nb + j] = npart[2 * qq][u] + npart[2 * qq + 1][u];
  }
}

struct SelPtrs {
  int nb, ncand, words, ld;  // key blocks (columns), candidate key blocks, mask words, row stride
  int nq, nqc;               // query blocks (rows), candidate query blocks
  const float *qbar, *kbar, *ztil;
  float *ytil, *gtil, *P, *q, *t, *K, *G, *J, *Jbest, *J0;
  uint32_t *dmask, *bmask;
  uint32_t* asplit;      // bf16x2 [3][H][nb][32]: g~ as three bf16 terms (tensor-core gains)
  float* cdot;           // [H, nb] y~_i . g~_i
  int64_t split_stride;  // H nb 32: uint32 words per term
  int32_t* kcount;       // [H, nq] key blocks kept by each candidate row
  uint32_t* status;      // device status word (first error wins)
};

__host__ __device__ inline SelPtrs sel_ptrs(const Shape& s, char* ws, const ress_ws_layout& L) {
  SelPtrs p;
  p.nb = s.nb;
  p.ncand = s.ncand;
  p.nq = s.nq;
  p.nqc = s.nqc;
  p.words = s.words;
  p.ld = s.ld;
  p.qbar = (const float*)(ws + L.qbar);
  p.kbar = (const float*)(ws + L.kbar);
  p.ztil = (const float*)(ws + L.ztil);
  p.ytil = (float*)(ws + L.ytil);
  p.gtil = (float*)(ws + L.gtil);
  p.P = (float*)(ws + L.P);
  p.q = (float*)(ws + L.q);
  p.t = (float*)(ws + L.t);
  p.K = (float*)(ws + L.K);
  p.G = (float*)(ws + L.G);
  p.J = (float*)(ws + L.J);
  p.Jbest = (float*)(ws + L.Jbest);
  p.J0 = (float*)(ws + L.J0);
  p.dmask = (uint32_t*)(ws + L.dmask);
  p.bmask = (uint32_t*)(ws + L.bmask);
  p.asplit = (uint32_t*)(ws + L.asplit);
  p.cdot = (float*)(ws + L.cdot);
  p.split_stride = (int64_t)s.H * s.nq * 32;
  p.kcount = (int32_t*)(ws + L.kcount);
  p.status = (uint32_t*)(ws + L.status);
  return p;
}

// Square root by the SFU (sqrt.approx: a few ulp, against the IEEE-rounded sqrtf's longer
// sequence); q >= 0 here, and sqrt of 0 is 0.
__device__ __forceinline__ float sqrt_approx(float x) {
  float y;
  asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Order-preserving map of a float to uint32; every non-NaN value maps above 0, so 0 can
// mark "not a candidate".  -0 is folded onto +0; NaN maps to the lowest candidate value.
__device__ __forceinline__ uint32_t order_key(float x) {
  x = x + 0.0f;
  const uint32_t b = __float_as_uint(x);
  if (x != x) return 1u;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// ------------------------------------------------------------------------------------
// Exact top-m for one warp over keys kk[0..n) in shared memory (block j has key kk[j]):
// the m largest keys, ties to the lower block index (the order the oracle uses).  With
// `member` set, only blocks whose bit in member[] equals `want` take part.  Result: the
// chosen blocks' bits in sel[words] (cleared first).
//
// 1. lower bound: the m-th largest value among every lane's local top-ceil(m/32) keys is
//    <= the m-th largest key overall (those 32 ceil(m/32) values include m entries);
// 2. survivors: the participating keys >= that bound (usually about 1.5 m of them) are
//    compacted, in block order, into a short list;
// 3. the m-th largest survivor T is found by a radix select over the survivors (8-bit
//    digits; select_radix), or bit by bit without radix counters (select_exact), and the
//    survivors > T plus the lowest-index ones == T are chosen.
// When m needs more than kTopK candidates per lane, or too many keys tie at the bound,
// step 3 runs bit by bit on all participating keys instead (same result, slower).  The
// restoration rounds use warp_topm_pair below, which selects on both sides of the drop set
// at once.
// ------------------------------------------------------------------------------------
constexpr int kTopK = 4;          // lane-local candidates: fast path for m <= 128
constexpr int kSurvivors = 256;   // capacity of the survivor list

__device__ __forceinline__ bool takes_part(const uint32_t* member, bool want, int j) {
  return member == nullptr || (((member[j >> 5] >> (j & 31)) & 1u) != 0) == want;
}

// m-th largest of the values v[] (up to N per lane), bit by bit with early exit.
template <int N>
__device__ __forceinline__ uint32_t mth_largest(const uint32_t (&v)[N], int m) {
  uint32_t lo = 0;
  for (int bit = 31; bit >= 0; --bit) {
    const uint32_t cand = lo | (1u << bit);
    int cnt = 0;
#pragma unroll
    for (int k = 0; k < N; ++k) cnt += v[k] >= cand ? 1 : 0;
    cnt = __reduce_add_sync(kFull, cnt);
    if (cnt >= m) {
      lo = cand;
      if (cnt == m) break;
    }
  }
  return lo;
}

// Exact selection over a list of n (key, index) pairs in ascending index order; with `member`
// the list is kk itself (index = position) filtered by membership, otherwise (sk, si).
__device__ void select_exact(const uint32_t* keys, const uint16_t* idx, int n, int m,
                             const uint32_t* member, bool want, uint32_t* sel) {
  const int lane = threadIdx.x & 31;
  auto part = [&](int x) { return idx != nullptr || takes_part(member, want, x); };
  uint32_t lo = 0;
  for (int bit = 31; bit >= 0; --bit) {
    const uint32_t cand = lo | (1u << bit);
    int cnt = 0;
#pragma unroll 4
    for (int x = lane; x < n; x += 32) cnt += (keys[x] >= cand && part(x)) ? 1 : 0;
    cnt = __reduce_add_sync(kFull, cnt);
    if (cnt >= m) {
      lo = cand;
      if (cnt == m) break;
    }
  }
  int gt = 0;
#pragma unroll 4
  for (int x = lane; x < n; x += 32) gt += (keys[x] > lo && part(x)) ? 1 : 0;
  gt = __reduce_add_sync(kFull, gt);
  const int need = m - gt;
  int taken = 0;
  for (int x0 = 0; x0 < n; x0 += 32) {
    const int x = x0 + lane;
    const bool in = x < n && part(x);
    const uint32_t v = in ? keys[x] : 0u;
    const bool is_eq = in && v == lo;
    const uint32_t eqb = __ballot_sync(kFull, is_eq);
    const int rank = taken + __popc(eqb & ((1u << lane) - 1u));
    if ((in && v > lo) || (is_eq && rank < need)) {
      const int j = idx ? (int)idx[x] : x;
      atomicOr(&sel[j >> 5], 1u << (j & 31));
    }
    taken += __popc(eqb);
  }
}

// A chosen block: bit j of the bitmask sel, or entry `pos` of the list lst as j | flag.
__device__ __forceinline__ void choose_block(uint32_t* sel, uint16_t* lst, uint16_t flag, int j,
                                             int pos) {
  if (lst)
    lst[pos] = (uint16_t)(j | flag);
  else
    atomicOr(&sel[j >> 5], 1u << (j & 31));
}

// Exact selection over a survivor list (keys[0..n) with block indices idx[], in ascending
// index order): the m largest keys, ties to the lower index, by a most-significant-first
// radix select with 8-bit digits whose 256 counters live in `hist` (per-warp shared
// scratch, 16-byte aligned).  Each pass fixes one byte of the m-th largest key and stops
// early once the keys that share the fixed bytes are exactly the ones still needed; a final
// pass in index order takes the keys above that prefix and the first `need` equal to it.
// The chosen blocks go to the bitmask sel, or, with lst set, to lst[0..m) as j | flag (in an
// order fixed by the data, so that sums over the list are reproducible).
__device__ void select_radix(const uint32_t* keys, const uint16_t* idx, int n, int m,
                             uint32_t* hist, uint32_t* sel, uint16_t* lst = nullptr,
                             uint16_t flag = 0) {
  const int lane = threadIdx.x & 31;
  if (n <= m) {  // every survivor is chosen
    for (int x = lane; x < n; x += 32) choose_block(sel, lst, flag, (int)idx[x], x);
    return;
  }
  if (n <= 32) {
    // one survivor per lane: a bitonic sort of (key, lower index first) composites,
    // descending; lanes 0..m-1 then hold the chosen blocks
    unsigned long long c = 0ull;  // below every survivor (keys are >= 1)
    if (lane < n) c = ((unsigned long long)keys[lane] << 32) | (0xffffu - (uint32_t)idx[lane]);
#pragma unroll
    for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
      for (int j = k >> 1; j >= 1; j >>= 1) {
        const unsigned long long o = __shfl_xor_sync(kFull, c, j);
        const bool keep_max = ((lane & k) == 0) == ((lane & j) == 0);
        c = keep_max ? (c > o ? c : o) : (c < o ? c : o);
      }
    }
    if (lane < m) choose_block(sel, lst, flag, 0xffff - (int)(c & 0xffffu), lane);
    return;
  }
  uint32_t prefix = 0u, pmask = 0u;
  int need = m;  // keys still to choose among those matching the prefix
  uint4* h4 = reinterpret_cast<uint4*>(hist);
  // bytes above the highest bit in which the survivors differ are common to all: start
  // below them
  uint32_t diff = 0u;
  for (int x = lane; x < n; x += 32) diff |= keys[x] ^ keys[0];
  diff = __reduce_or_sync(kFull, diff);
  const int top_shift = diff ? (31 - __clz(diff)) / 8 * 8 : 0;
  if (top_shift < 24) {
    pmask = 0xffffffffu << (top_shift + 8);
    prefix = keys[0] & pmask;
  }
  for (int shift = top_shift; shift >= 0; shift -= 8) {
    h4[2 * lane] = make_uint4(0u, 0u, 0u, 0u);
    h4[2 * lane + 1] = make_uint4(0u, 0u, 0u, 0u);
    __syncwarp();
    for (int x = lane; x < n; x += 32) {
      const uint32_t k = keys[x];
      if ((k & pmask) == prefix) atomicAdd(&hist[(k >> shift) & 255u], 1u);
    }
    __syncwarp();
    // lane l owns digits base + 7 .. base, base = 8 (31 - l): lane 0 the highest
    const int base = 8 * (31 - lane);
    const uint4 lo4 = h4[2 * (31 - lane)], hi4 = h4[2 * (31 - lane) + 1];
    const uint32_t c[8] = {hi4.w, hi4.z, hi4.y, hi4.x, lo4.w, lo4.z, lo4.y, lo4.x};
    int sum = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) sum += (int)c[i];
    int inc = sum;  // inclusive count over lanes 0..l (digits above and at this lane's)
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, inc, o);
      if (lane >= o) inc += y;
    }
    const int exc = inc - sum;
    const uint32_t who = __ballot_sync(kFull, exc < need && need <= inc);
    const int src = __ffs(who) - 1;
    int digit = 0, before = 0, cnt = 0;
    if (lane == src) {
      int run = exc;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        if (cnt == 0 && run + (int)c[i] >= need) {
          digit = base + 7 - i;
          before = run;
          cnt = (int)c[i];
        }
        run += (int)c[i];
      }
    }
    digit = __shfl_sync(kFull, digit, src);
    before = __shfl_sync(kFull, before, src);
    cnt = __shfl_sync(kFull, cnt, src);
    need -= before;
    prefix |= (uint32_t)digit << shift;
    pmask |= 255u << shift;
    if (cnt == need) break;  // every key with this prefix is chosen
  }
  int taken = 0, out = 0;
  const uint32_t below = (1u << lane) - 1u;
  for (int x0 = 0; x0 < n; x0 += 32) {
    const int x = x0 + lane;
    const bool in = x < n;
    const uint32_t v = in ? (keys[x] & pmask) : 0u;
    const bool is_eq = in && v == prefix;
    const uint32_t eqb = __ballot_sync(kFull, is_eq);
    const int rank = taken + __popc(eqb & below);
    const bool chosen = (in && v > prefix) || (is_eq && rank < need);
    const uint32_t cb = __ballot_sync(kFull, chosen);
    if (chosen) choose_block(sel, lst, flag, (int)idx[x], out + __popc(cb & below));
    taken += __popc(eqb);
    out += __popc(cb);
  }
}

// The lower bound of step 1 with KT = ceil(m / 32) keys kept per lane: the m-th largest of
// the lanes' KT largest participating keys.
template <int KT>
__device__ __forceinline__ uint32_t lane_topk_bound(const uint32_t* kk, int n, int m,
                                                    const uint32_t* member, bool want) {
  const int lane = threadIdx.x & 31;
  uint32_t top[KT];
#pragma unroll
  for (int k = 0; k < KT; ++k) top[k] = 0u;
#pragma unroll 2
  for (int x = lane; x < n; x += 32) {
    uint32_t v = takes_part(member, want, x) ? kk[x] : 0u;
#pragma unroll
    for (int k = 0; k < KT; ++k) {
      const uint32_t hi = max(top[k], v);
      v = min(top[k], v);
      top[k] = hi;
    }
  }
  return mth_largest(top, m);
}

// Requires m <= number of participating blocks.  sk/si: survivor scratch (kSurvivors);
// hist: 256 words for select_radix on the survivors (NULL: bit-by-bit select_exact).
__device__ void warp_topm(const uint32_t* kk, int n, int m, uint32_t* sel, int words,
                          uint32_t* sk, uint16_t* si, const uint32_t* member = nullptr,
                          bool want = true, uint32_t* hist = nullptr) {
  const int lane = threadIdx.x & 31;
  for (int w = lane; w < words; w += 32) sel[w] = 0u;
  __syncwarp();
  if (m <= 0) return;
  const int K = (m + 31) / 32;
  if (K > kTopK) {
    select_exact(kk, nullptr, n, m, member, want, sel);
    __syncwarp();
    return;
  }
  // 1. lane-local top-K (descending) of the participating keys, then the lower bound
  uint32_t bound;
  switch (K) {
    case 1: bound = lane_topk_bound<1>(kk, n, m, member, want); break;
    case 2: bound = lane_topk_bound<2>(kk, n, m, member, want); break;
    case 3: bound = lane_topk_bound<3>(kk, n, m, member, want); break;
    default: bound = lane_topk_bound<4>(kk, n, m, member, want); break;
  }
  // 2. survivors (participating, >= bound), compacted in block order
  int cnt = 0;
  for (int x0 = 0; x0 < n; x0 += 32) {
    const int x = x0 + lane;
    const bool keep = x < n && kk[x] >= bound && takes_part(member, want, x);
    const uint32_t b = __ballot_sync(kFull, keep);
    const int pos = cnt + __popc(b & ((1u << lane) - 1u));
    if (keep && pos < kSurvivors) {
      sk[pos] = kk[x];
      si[pos] = (uint16_t)x;
    }
    cnt += __popc(b);
  }
  __syncwarp();
  // 3. exact selection on the survivors (or on every participating key if they overflowed)
  if (cnt > kSurvivors)
    select_exact(kk, nullptr, n, m, member, want, sel);
  else if (hist)
    select_radix(sk, si, cnt, m, hist, sel);
  else
    select_exact(sk, si, cnt, m, nullptr, true, sel);
  __syncwarp();
}

// This lane's two largest keys on each side of a drop set, kept while the keys are written.
struct LaneTop2 {
  uint32_t d1 = 0, d2 = 0, b1 = 0, b2 = 0;  // in D: largest, second; outside D: same
  __device__ __forceinline__ void add(uint32_t v, bool inD) {
    uint32_t& a1 = inD ? d1 : b1;
    uint32_t& a2 = inD ? d2 : b2;
    a2 = max(a2, min(a1, v));
    a1 = max(a1, v);
  }
};

// The m-th largest (1 <= m <= 64) of the 64 values held two per lane (element 2 lane + s
// holds v[s]): a bitonic sort of the 64 values across the warp, descending.
__device__ __forceinline__ uint32_t mth_of_64(uint32_t a, uint32_t b, int m) {
  const int lane = threadIdx.x & 31;
  uint32_t v[2] = {a, b};
#pragma unroll
  for (int k = 2; k <= 64; k <<= 1) {
#pragma unroll
    for (int j = k >> 1; j >= 1; j >>= 1) {
      if (j == 1) {  // the partner is the lane's other element
        const bool desc = ((2 * lane) & k) == 0;
        const uint32_t hi = max(v[0], v[1]), lo = min(v[0], v[1]);
        v[0] = desc ? hi : lo;
        v[1] = desc ? lo : hi;
      } else {
#pragma unroll
        for (int s = 0; s < 2; ++s) {
          const int e = 2 * lane + s;
          const uint32_t o = __shfl_xor_sync(kFull, v[s], j >> 1);
          // in a descending run the lower element of a pair keeps the larger value
          v[s] = (((e & k) == 0) == ((e & j) == 0)) ? max(v[s], o) : min(v[s], o);
        }
      }
    }
  }
  const uint32_t mine = ((m - 1) & 1) ? v[1] : v[0];
  return __shfl_sync(kFull, mine, (m - 1) >> 1);
}

// Both selections of a restoration round at once, for m <= 64: the m largest keys among
// the blocks in D (bit set in Dw) into selD and the m largest among the other candidates
// into selB, ties to the lower block index.  `top` holds this lane's two largest keys on
// each side (0 where it has none), taken while the keys were written, so the lane-local
// pass of warp_topm is not needed: the m-th largest of the 64 lane values of a side (a
// bitonic sort across the warp) bounds that side's m-th key from below.  Both survivor
// lists come from one pass (four blocks per lane and step, one warp scan for the store
// positions); each side then selects exactly (radix select on its survivors).
// Returns true when the chosen blocks went to lst (restores at lst[0..m), drops at
// lst[m..2m) with bit 15 set) instead of the bitmasks; lst lies in the key area after its
// first 256 words (the radix counters).
__device__ bool warp_topm_pair(const uint32_t* kk, int n, int m, const uint32_t* Dw,
                               const LaneTop2& top, uint32_t* selD, uint32_t* selB,
                               int words, uint32_t* sk, uint16_t* si, uint16_t* lst) {
  const int lane = threadIdx.x & 31;
  for (int w = lane; w < words; w += 32) selD[w] = selB[w] = 0u;
  __syncwarp();
  if (m <= 0) return false;
  // the m-th largest of the 64 lane values of a side bounds that side's m-th key from below
  const uint32_t bD = mth_of_64(top.d1, top.d2, m), bB = mth_of_64(top.b1, top.b2, m);
  constexpr int kHalf = kSurvivors / 2;
  int cntD = 0, cntB = 0;
  // survivors in ascending block order, four consecutive blocks per lane and step: each
  // lane's counts on both sides (packed) go through one warp scan for the store positions
  for (int x0 = 0; x0 < n; x0 += 128) {
    const int x = x0 + 4 * lane;
    uint32_t fD = 0u, fB = 0u;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (x < n) {
      v = *reinterpret_cast<const uint4*>(kk + x);  // 16-byte aligned, inside the key area
      const uint32_t dbits = Dw[x >> 5] >> (x & 31);
      const uint32_t k4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (x + u < n) {
          const bool inD = (dbits >> u) & 1u;
          if (inD && k4[u] >= bD) fD |= 1u << u;
          if (!inD && k4[u] >= bB) fB |= 1u << u;
        }
      }
    }
    const int c = __popc(fD) | (__popc(fB) << 16);
    int inc = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, inc, o);
      if (lane >= o) inc += y;
    }
    const int total = __shfl_sync(kFull, inc, 31);
    if (fD | fB) {
      int pD = cntD + ((inc - c) & 0xffff), pB = cntB + ((inc - c) >> 16);
      const uint32_t k4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if ((fD >> u) & 1u) {
          if (pD < kHalf) {
            sk[pD] = k4[u];
            si[pD] = (uint16_t)(x + u);
          }
          ++pD;
        }
        if ((fB >> u) & 1u) {
          if (pB < kHalf) {
            sk[kHalf + pB] = k4[u];
            si[kHalf + pB] = (uint16_t)(x + u);
          }
          ++pB;
        }
      }
    }
    cntD += total & 0xffff;
    cntB += total >> 16;
  }
  __syncwarp();
  if (cntD <= kHalf && cntB <= kHalf) {
    // the keys are no longer needed: their first 256 words hold the radix counters
    select_radix(sk, si, cntD, m, const_cast<uint32_t*>(kk), selD, lst, 0);
    select_radix(sk + kHalf, si + kHalf, cntB, m, const_cast<uint32_t*>(kk), selB, lst + m, 0x8000);
    __syncwarp();
    return true;
  }
  if (cntD > kHalf)
    select_exact(kk, nullptr, n, m, Dw, true, selD);
  else
    select_exact(sk, si, cntD, m, nullptr, true, selD);
  if (cntB > kHalf)
    select_exact(kk, nullptr, n, m, Dw, false, selB);
  else
    select_exact(sk + kHalf, si + kHalf, cntB, m, nullptr, true, selB);
  __syncwarp();
  return false;
}

// g~ of row ri (this lane's channels 2 lane, 2 lane + 1), its three bf16 terms (the A
// operands of the tensor-core gains) and c_i = y~_i . g~_i.
__device__ __forceinline__ void store_gtil(const SelPtrs& p, int64_t ri, int lane, float2 y,
                                           float g0, float g1) {
  *reinterpret_cast<float2*>(p.gtil + ri * 64 + 2 * lane) = make_float2(g0, g1);
  uint32_t hi, mid, lo;
  split3_bf16x2(g0, g1, hi, mid, lo);
  uint32_t* gs = p.asplit + ri * 32 + lane;
  gs[0] = hi;
  gs[p.split_stride] = mid;
  gs[2 * p.split_stride] = lo;
  const float c = warp_sum(y.x * g0 + y.y * g1);
  if (lane == 0) p.cdot[ri] = c;
}

// Bits of word w that are valid key blocks (< nb).
__device__ __forceinline__ uint32_t valid_bits(int w, int n) {
  const int rem = n - w * 32;
  return rem >= 32 ? kFull : (rem <= 0 ? 0u : ((1u << rem) - 1u));
}

// g~ = sum_{j not in D} P_ij (z~_j - y~_i) and K = sum_{j not in D} P_ij for one row, by
// one warp (lane owns channels 2*lane, 2*lane+1), in ascending j.  The kept blocks are
// first compacted into idx[] (per-warp shared memory, >= nb entries) so that the loads of
// eight blocks are in flight together.
__device__ __forceinline__ void kept_drift(const uint32_t* D, const SelPtrs& p,
                                           const float* __restrict__ Prow,
                                           const float* __restrict__ zt, float y0, float y1,
                                           uint32_t* idx, float& g0, float& g1, float& K) {
  const int lane = threadIdx.x & 31;
  // lane l compacts mask word w0 + l: one warp scan of the words' kept counts gives each
  // word's first list position, then each lane writes its own word's blocks (ascending)
  int n = 0;
  for (int w0 = 0; w0 < p.words; w0 += 32) {
    const int w = w0 + lane;
    uint32_t keep = w < p.words ? ~D[w] & valid_bits(w, p.nb) : 0u;
    const int c = __popc(keep);
    int inc = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, inc, o);
      if (lane >= o) inc += y;
    }
    for (int pos = n + inc - c; keep; keep &= keep - 1u, ++pos) idx[pos] = w * 32 + __ffs(keep) - 1;
    n += __shfl_sync(kFull, inc, 31);
  }
  __syncwarp();
  g0 = g1 = K = 0.f;
  for (int k0 = 0; k0 < n; k0 += 8) {
    float pj[8];
    float2 z[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      if (k0 + u < n) {
        const int j = idx[k0 + u];
        pj[u] = Prow[j];
        z[u] = *reinterpret_cast<const float2*>(zt + (int64_t)j * 64 + 2 * lane);
      }
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      if (k0 + u < n) {
        // g += P_j (z~_j - y~), both channels in packed instructions (z - y as an exact
        // fma with 1, so the bits are those of the scalar form)
        float d0, d1;
        ptx::fma2(d0, d1, z[u].x, z[u].y, 1.0f, 1.0f, -y0, -y1);
        ptx::fma2(g0, g1, pj[u], pj[u], d0, d1, g0, g1);
        K += pj[u];
      }
    }
  }
  __syncwarp();
}

// The state after a round from the one before it: the restored blocks R join the kept set
// and the dropped blocks X leave it, so g~ += sum_R P_k (z~_k - y~) - sum_X P_k (z~_k - y~)
// and K += sum_R P_k - sum_X P_k over the 2m swapped blocks (exactly the kept-set sums of
// Eq. 10-11 in exact arithmetic), taken in the order of their list (j | 0x8000 for a
// dropped block).  Same lane layout and staging as kept_drift.
__device__ __forceinline__ void swap_drift_list(const uint16_t* lst, int n,
                                                const float* __restrict__ Prow,
                                                const float* __restrict__ zt, float y0, float y1,
                                                float& g0, float& g1, float& K) {
  const int lane = threadIdx.x & 31;
  for (int k0 = 0; k0 < n; k0 += 8) {
    float pj[8];
    float2 z[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      pj[u] = 0.f;
      z[u] = make_float2(y0, y1);
      if (k0 + u < n) {
        const uint32_t e = lst[k0 + u];
        const int j = (int)(e & 0x7fffu);
        const float pv = Prow[j];
        pj[u] = (e >> 15) ? -pv : pv;
        z[u] = *reinterpret_cast<const float2*>(zt + (int64_t)j * 64 + 2 * lane);
      }
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      g0 = fmaf(pj[u], z[u].x - y0, g0);
      g1 = fmaf(pj[u], z[u].y - y1, g1);
      K += pj[u];
    }
  }
  __syncwarp();
}

// Per-warp scratch of the per-row kernels: keys [key_words(ld)] u32, survivor keys
// [kSurvivors] u32, survivor indices [kSurvivors] u16, bitmask words (and, in the score
// kernel, 256 radix counters after them).
// The key area holds at least 320 words, so that once the keys are spent it can hold the
// 256 radix counters and a list of up to 128 swapped blocks (u16); the total is a multiple
// of 4 words (16-byte aligned per-warp areas).
__host__ __device__ constexpr int key_words(int ld) { return ld > 320 ? ld : 320; }
__host__ __device__ constexpr size_t warp_scratch_words(int ld, int words_per_warp) {
  return ((size_t)key_words(ld) + kSurvivors + kSurvivors / 2 + words_per_warp + 3) / 4 * 4;
}
// the score kernel's words after the survivors: its drop-set mask, then (with the CDF rule,
// which keeps the keys past the selection) 256 radix counters
__host__ __device__ constexpr int score_mask_words(int words, bool cdf) {
  return (words + 3) / 4 * 4 + (cdf ? 256 : 0);
}




// Exact decrease of J (Eq. 16) when G changes by dG and K by u, with the denominators
// clamped at eps as in Eq. 7.  The two fractions are combined over one denominator so that
// the result carries no cancellation of J-sized terms, and no branch is taken per block.
__device__ __forceinline__ float delta_J(float G, float K, float dG, float u) {
  // G / Kc^2 - (G + dG) / K2c^2 = (G (K2c - Kc)(K2c + Kc) - dG Kc^2) / (Kc^2 K2c^2), with
  // Kc = max(K, eps) and K2c = max(K + u, eps); K2c - Kc is u when no clamp applies
  const float Kc = fmaxf(K, kEps), K2c = fmaxf(K + u, kEps);
  const float KK = Kc * Kc;
  const float num = fmaf(G * (K2c - Kc), K2c + Kc, -dG * KK);
  return __fdividef(num, KK * (K2c * K2c));
}


// ------------------------------------------------------------------------------------
// Per-row kernels: one warp per candidate query row, 4 rows per CTA.  They hold few
// registers so that many warps share an SM and hide the latency of the row's loads.
// ------------------------------------------------------------------------------------
constexpr int kRowWarps = 4;

// Candidate keys of one row, four blocks per lane and load (rows are 16-byte aligned and
// padded to a multiple of 32 entries).
template <typename KeyFn>
__device__ __forceinline__ void row_keys(int n, uint32_t* kk, KeyFn key_of) {
  const int lane = threadIdx.x & 31;
#pragma unroll 2
  for (int j4 = 4 * lane; j4 < n; j4 += 128) {
    uint32_t k4[4];
    key_of(j4, k4);
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (j4 + u < n) kk[j4 + u] = k4[u];
  }
  __syncwarp();
}

// SplitMix64 (Steele, Lea and Flood, OOPSLA 2014) at state x: advance by the golden-ratio
// increment, then that paper's mix.  The random selection keys of the ablation variant.
__device__ __forceinline__ unsigned long long splitmix64(unsigned long long x) {
  unsigned long long z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// CDF threshold (Table 3, the top-p rule of probability-based selection): after the c_h
// largest keys a row keeps further candidates in key order (ties to the lower index) until
// the pooled mass of its kept blocks, the always-kept ones included, reaches tau.  kk holds
// the candidates' keys and D the drop set (the candidates not yet kept).  The blocks that
// join are the shortest prefix of D in key order whose mass reaches tau - (kept mass); it
// is found without sorting: bit by bit, the largest key T such that the mass of the blocks
// of D with key >= T still reaches that need, then, among the blocks whose key is exactly T,
// the shortest prefix by index.  Each pass sums per lane in ascending j and then across the
// warp in a fixed order, so a pass's sum never decreases when its set grows.
__device__ void cdf_extend(const uint32_t* kk, const float* __restrict__ Prow, uint32_t* D,
                           int ncand, int nb, int words, float tau) {
  const int lane = threadIdx.x & 31;
  auto in_D = [&](int j) { return ((D[j >> 5] >> (j & 31)) & 1u) != 0u; };
  float kept = 0.f;
  for (int j = lane; j < nb; j += 32)
    if (!in_D(j)) kept += Prow[j];
  const float need = tau - warp_sum(kept);
  if (!(need > 0.f)) return;
  auto mass_from = [&](uint32_t T) {  // mass of the blocks of D with key >= T
    float s = 0.f;
    for (int j = lane; j < ncand; j += 32)
      if (in_D(j) && kk[j] >= T) s += Prow[j];
    return warp_sum(s);
  };
  uint32_t T = 0u;  // mass_from(T) >= need holds throughout, unless even all of D falls short
  int L = ncand;    // the blocks with key T and index <= L join
  if (mass_from(0u) >= need) {
    for (int bit = 31; bit >= 0; --bit) {
      const uint32_t cand = T | (1u << bit);
      if (mass_from(cand) >= need) T = cand;
    }
    // every block with key > T is needed (their mass alone falls short); the ties at T join
    // in ascending index until the rest of the need is met
    const float need_t = need - (T == 0xffffffffu ? 0.f : mass_from(T + 1u));
    auto tie_mass_below = [&](int x) {
      float s = 0.f;
      for (int j = lane; j < min(x, ncand); j += 32)
        if (in_D(j) && kk[j] == T) s += Prow[j];
      return warp_sum(s);
    };
    L = 0;  // the largest L with the ties below index L still short of need_t
    for (int bit = 12; bit >= 0; --bit) {
      const int cand = L | (1 << bit);
      if (cand <= ncand && tie_mass_below(cand) < need_t) L = cand;
    }
  }
  for (int w = 0; w < words; ++w) {
    const int j = w * 32 + lane;
    const bool joins =
        j < ncand && in_D(j) && (kk[j] > T || (kk[j] == T && j <= L));
    const uint32_t m = __ballot_sync(kFull, joins);
    __syncwarp();
    if (lane == 0) D[w] &= ~m;
    __syncwarp();
  }
}

// Initial selection (Eq. 7) and the state of Eq. 10-12.  grid (ceil(|P| / 4), H).
// The variant picks the key: the Eq. 7 drift key (ReSS), the pooled probability, or the top
// 24 bits of SplitMix64 at seed + (h 4096 + i) 4096 + j; the full sign flip keeps the
// smallest keys (complemented keys, ties still to the lower index).
// KEY: the key variant (v.key), a template parameter so that the per-block key has no branch.
template <int KEY>
__global__ void __launch_bounds__(32 * kRowWarps, 9) k_score_rows(SelPtrs p, Budgets bud,
                                                                  Variant v) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y, i = blockIdx.x * kRowWarps + warp;
  if (i >= p.nqc) return;
  const int64_t ri = (int64_t)h * p.nq + i;
  const float* Prow = p.P + ri * p.ld;
  const float* qrow = p.q + ri * p.ld;
  const float* zt_h = p.ztil + (int64_t)h * p.nb * 64;
  uint32_t* base = reinterpret_cast<uint32_t*>(smem_raw) +
                   (size_t)warp * warp_scratch_words(p.ld, score_mask_words(p.words, v.cdf > 0.f));
  uint32_t* kk = base;
  uint32_t* sk = base + key_words(p.ld);
  uint16_t* si = reinterpret_cast<uint16_t*>(sk + kSurvivors);
  uint32_t* sel = sk + kSurvivors + kSurvivors / 2;
  // radix counters: in the spent key area, or after the mask when the CDF rule needs the keys
  uint32_t* hist = v.cdf > 0.f ? sel + (p.words + 3) / 4 * 4 : kk;
  row_keys(p.ncand, kk, [&](int j, uint32_t (&k4)[4]) {
    const float4 P4 = *reinterpret_cast<const float4*>(Prow + j);
    const float4 q4 = *reinterpret_cast<const float4*>(qrow + j);
    const float pv[4] = {P4.x, P4.y, P4.z, P4.w}, qv[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      uint32_t key;
      if (KEY == 0)  // s_ij / max(1 - P_ij, eps), s_ij = P_ij sqrt(q_ij); the SFU's square root
        key = order_key(__fdividef(pv[u] * sqrt_approx(qv[u]), fmaxf(1.0f - pv[u], kEps)));
      else if (KEY == 1)
        key = order_key(pv[u]);
      else
        key = (uint32_t)(splitmix64(v.seed + ((unsigned long long)h * 4096ull + (unsigned long long)i) *
                                                 4096ull + (unsigned long long)(j + u)) >> 40) + 1u;
      k4[u] = (v.direction == 2) ? ~key : key;
    }
  });
  warp_topm(kk, p.ncand, bud.c[h], sel, p.words, sk, si, nullptr, true, hist);  // sel = kept
  // drop set D0 = candidates not kept
  for (int w = lane; w < p.words; w += 32) sel[w] = valid_bits(w, p.ncand) & ~sel[w];
  __syncwarp();
  if (v.cdf > 0.f) cdf_extend(kk, Prow, sel, p.ncand, p.nb, p.words, v.cdf);
  int ndrop = 0;
  for (int w = lane; w < p.words; w += 32) {
    const uint32_t d = sel[w];
    p.dmask[ri * p.words + w] = d;
    p.bmask[ri * p.words + w] = d;
    ndrop += __popc(d);
  }
  ndrop = __reduce_add_sync(kFull, ndrop);
  if (lane == 0) p.kcount[ri] = p.nb - ndrop;
  __syncwarp();
  const float2 y = *reinterpret_cast<const float2*>(p.ytil + ri * 64 + 2 * lane);
  float g0, g1, K;
  kept_drift(sel, p, Prow, zt_h, y.x, y.y, kk, g0, g1, K);
  const float G = warp_sum(g0 * g0 + g1 * g1);
  const float Kc = fmaxf(K, kEps);
  const float J = G / (Kc * Kc);
  store_gtil(p, ri, lane, y, g0, g1);
  if (lane == 0) {
    p.K[ri] = K;
    p.G[ri] = G;
    p.J[ri] = J;
    p.Jbest[ri] = J;
    p.J0[ri] = J;
  }
}

// ------------------------------------------------------------------------------------
// Restoration round r (Sec. 4.3, Eq. 13-17).  The gain inner products t_ij of the round
// come from k_dot (tensor cores, k_dot.cu); the rest of the round runs per row here.
// ------------------------------------------------------------------------------------
// Restoration round r, per row: exact top-m restores and drops from the round-start state,
// update, track-best.  grid (ceil(|P| / 4), H).  With a maximising variant the keys are the
// increases of J and track-best keeps the largest J.
// MAXIMIZE: a maximising variant (keys are the increases of J, track-best keeps the largest
// J), a template parameter so that the per-block key has no select.
template <int MAXIMIZE>
__global__ void __launch_bounds__(32 * kRowWarps, 10) k_round_rows(SelPtrs p, Budgets bud,
                                                                  int round, float rho) {
  constexpr bool maximize = MAXIMIZE != 0;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y, i = blockIdx.x * kRowWarps + warp;
  const int m = swap_count(bud.c[h], p.ncand, round, rho);
  if (m <= 0 || i >= p.nqc) return;
  const int64_t ri = (int64_t)h * p.nq + i;
  const float* Prow = p.P + ri * p.ld;
  const float* qrow = p.q + ri * p.ld;
  const float* trow = p.t + ri * p.ld;
  const float* zt_h = p.ztil + (int64_t)h * p.nb * 64;
  uint32_t* base = reinterpret_cast<uint32_t*>(smem_raw) + (size_t)warp * warp_scratch_words(p.ld, 3 * p.words);
  uint32_t* kk = base;
  uint32_t* sk = base + key_words(p.ld);
  uint16_t* si = reinterpret_cast<uint16_t*>(sk + kSurvivors);
  uint32_t* Dw = sk + kSurvivors + kSurvivors / 2;  // current drop set
  uint32_t* Rw = Dw + p.words;                       // chosen restores
  uint32_t* Xw = Rw + p.words;                       // chosen drops
  for (int w = lane; w < p.words; w += 32) Dw[w] = p.dmask[ri * p.words + w];
  const float K = p.K[ri], G = p.G[ri];
  __syncwarp();
  LaneTop2 top;  // this lane's two largest keys in D and outside it
  // one pass over the candidates: a block k in D is a restore candidate (u = +P_k,
  // dG = -2 P_k t_k + P_k^2 q_k, Eq. 13-14), a kept candidate a drop candidate (u = -P_k,
  // dG = +2 P_k t_k + P_k^2 q_k, Eq. 15); the key is the exact decrease of J (Eq. 16)
  row_keys(p.ncand, kk, [&](int j, uint32_t (&k4)[4]) {
    const float4 P4 = *reinterpret_cast<const float4*>(Prow + j);
    const float4 q4 = *reinterpret_cast<const float4*>(qrow + j);
    const float4 t4 = *reinterpret_cast<const float4*>(trow + j);
    const float pv[4] = {P4.x, P4.y, P4.z, P4.w}, qv[4] = {q4.x, q4.y, q4.z, q4.w},
                tv[4] = {t4.x, t4.y, t4.z, t4.w};
    const uint32_t dword = Dw[j >> 5] >> (j & 31);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const bool inD = (dword >> u) & 1u;
      const float s2 = pv[u] * pv[u] * qv[u];
      const float dG = inD ? fmaf(-2.0f * pv[u], tv[u], s2) : fmaf(2.0f * pv[u], tv[u], s2);
      const float dJ = delta_J(G, K, dG, inD ? pv[u] : -pv[u]);
      k4[u] = order_key(maximize ? -dJ : dJ);
      if (j + u < p.ncand) top.add(k4[u], inD);
    }
  });
  // the swapped blocks as a list: written by the selection itself on the common path
  // (after the radix counters in the key area), else gathered from the bitmasks R and X
  uint16_t* lst = reinterpret_cast<uint16_t*>(kk + 256);
  int nl = 2 * m;
  bool listed = false;
  if (m <= 64) {
    listed = warp_topm_pair(kk, p.ncand, m, Dw, top, Rw, Xw, p.words, sk, si, lst);
  } else {
    warp_topm(kk, p.ncand, m, Rw, p.words, sk, si, Dw, true);
    warp_topm(kk, p.ncand, m, Xw, p.words, sk, si, Dw, false);
  }
  if (round == 0) {
    // both selections took m blocks from their side only if the drop set holds that many on
    // each; a workspace whose drop set cannot give them (one the scoring did not write, or
    // one scored with other budgets) is reported instead of updated from.  Later rounds
    // read the drop sets this round wrote, whose sizes the swaps keep.
    int nd = 0;
    for (int w = lane; w < p.words; w += 32) nd += __popc(Dw[w] & valid_bits(w, p.ncand));
    nd = __reduce_add_sync(kFull, nd);
    if (nd < m || p.ncand - nd < m) {
      if (lane == 0) flag_status(p.status, kStatusBadRow);
      return;
    }
  }
  if (!listed) {
    lst = reinterpret_cast<uint16_t*>(kk);  // 2 key_words >= 2m entries
    nl = 0;
    for (int w = 0; w < p.words; ++w) {
      const uint32_t sw = Rw[w] | Xw[w];
      if ((sw >> lane) & 1u)
        lst[nl + __popc(sw & ((1u << lane) - 1u))] =
            (uint16_t)((w * 32 + lane) | (((Xw[w] >> lane) & 1u) << 15));
      nl += __popc(sw);
    }
    __syncwarp();
  }
  // every listed block changes sides: restores leave D, drops join it
  for (int e = lane; e < nl; e += 32) {
    const int j = lst[e] & 0x7fff;
    if (j < p.ncand) atomicXor(&Dw[j >> 5], 1u << (j & 31));
    else flag_status(p.status, kStatusBadIndex);
  }
  __syncwarp();
  // state of the new set (Eq. 10-12): the swapped blocks update g~ and K
  const float2 y = *reinterpret_cast<const float2*>(p.ytil + ri * 64 + 2 * lane);
  const float2 gold = *reinterpret_cast<const float2*>(p.gtil + ri * 64 + 2 * lane);
  float g0 = gold.x, g1 = gold.y, Kn = K;
  swap_drift_list(lst, nl, Prow, zt_h, y.x, y.y, g0, g1, Kn);
  const float Gn = warp_sum(g0 * g0 + g1 * g1);
  const float Kc = fmaxf(Kn, kEps);
  const float Jn = Gn / (Kc * Kc);
  const bool better = maximize ? (Jn > p.Jbest[ri]) : (Jn < p.Jbest[ri]);
  for (int w = lane; w < p.words; w += 32) {
    p.dmask[ri * p.words + w] = Dw[w];
    if (better) p.bmask[ri * p.words + w] = Dw[w];
  }
  store_gtil(p, ri, lane, y, g0, g1);
  if (lane == 0) {
    p.K[ri] = Kn;
    p.G[ri] = Gn;
    p.J[ri] = Jn;
    if (better) p.Jbest[ri] = Jn;
  }
}

// ------------------------------------------------------------------------------------
// Pairing of query blocks for the attention items (64-token grid, fixed budgets).  The
// attention runs two 64-row query blocks as one M = 128 tile over the union of their kept
// lists, so every key block kept by only one of them is half a tile of wasted tensor work.
// Within each window of kPairWindow candidate query blocks of a head, blocks are paired by
// the overlap of their best kept candidate sets, greedily by weight: of all pairs of
// unpaired blocks of the window, the one sharing most kept blocks is taken next (ties to
// the nearer pair, then to the lower first block).  Output: prow[h, 32 w + k] = a | b << 16 for the k-th pair of window
// w.  A row attends exactly its own kept blocks whichever block shares its tile; the partner
// decides only their order (the blocks kept by one of the two lead the list), so it moves a
// result by rounding alone.  grid (windows, H) x 512 threads: all warps form the
// window's overlaps, then take the pairs by weight (one block-wide maximum per pair).
// ------------------------------------------------------------------------------------
__global__ void __launch_bounds__(512) k_pairing(const uint32_t* __restrict__ bmask, int nq,
                                                 int words, int ncand, int npaired, int items,
                                                 int32_t* __restrict__ prow) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  constexpr int W = kPairWindow;
  // kept sets as rows of 64-bit words with an odd row stride, so that the eight rows one
  // load touches fall in distinct bank pairs
  const int words2 = (words + 1) >> 1, ks2 = words2 | 1;
  uint2* kept = reinterpret_cast<uint2*>(smem_raw);  // [W][ks2]
  const int h = blockIdx.y, w = blockIdx.x, t = threadIdx.x;
  const int r0 = W * w;
  const int n = min(W, 2 * npaired - r0);  // even
  if (n <= 0) return;
  for (int idx = t; idx < W * words2; idx += blockDim.x) {  // rows past n: empty
    const int r = idx / words2, wd = 2 * (idx - r * words2);
    uint2 v = make_uint2(0u, 0u);
    if (r < n) {
      const uint32_t* row = bmask + ((int64_t)h * nq + r0 + r) * words;
      v.x = ~row[wd] & valid_bits(wd, ncand);
      if (wd + 1 < words) v.y = ~row[wd + 1] & valid_bits(wd + 1, ncand);
    }
    kept[r * ks2 + (wd >> 1)] = v;
  }
  __syncthreads();
  // thread t: block a = t / 8 against the blocks g, g + 8, .., g + 56 (g = t mod 8); the
  // counts stay with the thread, which forms the keys of exactly these pairs below
  const int a = t >> 3, g = t & 7;
  int c[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) c[j] = 0;
  if (a < n) {
#pragma unroll 2
    for (int wd = 0; wd < words2; ++wd) {
      const uint2 ka = kept[a * ks2 + wd];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const uint2 kb = kept[(g + 8 * j) * ks2 + wd];
        c[j] += __popc(ka.x & kb.x) + __popc(ka.y & kb.y);
      }
    }
  }
  // Greedy matching by weight (the pair of unpaired blocks that shares most kept blocks
  // first; ties to the nearer pair, then to the lower first block), found in rounds: every
  // unpaired block points at its best unpaired partner, and blocks pointing at each other
  // are paired (the best remaining pair always is; 7 rounds on average at 32 views).  Eight
  // threads per block (thread t: block a = t / 8, partners g + 8 j, g = t mod 8).
  __shared__ int best_s[W], partner_s[W];
  __shared__ unsigned long long matched_s[2], lower_s[2];
  const int lane = t & 31;
  const uint32_t gmask = 0xFFu << (8 * (lane >> 3));  // the eight lanes of block a
  uint32_t key[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int b = g + 8 * j;
    const int d = b > a ? b - a : a - b, lo = min(a, b);
    // overlap < 2048 (clamped), |b - a| and min(a, b) < 64: one key per pair, every valid
    // key above 0; the pair's count is the same whichever of its blocks forms it
    key[j] = (b != a && b < n && a < n)
                 ? ((uint32_t)min(c[j], 2047) << 12) | ((uint32_t)(63 - d) << 6) | (uint32_t)(63 - lo)
                 : 0u;
  }
  if (t < W) partner_s[t] = -1;
  if (t < 2) matched_s[t] = 0ull;
  uint64_t freeb = n == 64 ? ~0ull : ((1ull << n) - 1ull);  // unpaired blocks of the window
  __syncthreads();
  for (int round = 0; round < W && __popcll(freeb) >= 2; ++round) {
    uint32_t k = 0u;
    if ((freeb >> a) & 1ull) {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if ((freeb >> (g + 8 * j)) & 1ull) k = max(k, key[j]);
    }
    k = __reduce_max_sync(gmask, k);
    if (g == 0) {
      const int d = 63 - (int)((k >> 6) & 63u), lo = 63 - (int)(k & 63u);
      best_s[a] = k == 0u ? -1 : (lo == a ? a + d : lo);
    }
    __syncthreads();
    if (g == 0 && ((freeb >> a) & 1ull)) {
      const int b = best_s[a];
      if (b >= 0 && best_s[b] == a) {
        partner_s[a] = b;
        atomicOr(&matched_s[round & 1], 1ull << a);
      }
    }
    __syncthreads();
    freeb &= ~matched_s[round & 1];
    if (t == 0) matched_s[(round + 1) & 1] = 0ull;  // read by every thread a round ago
  }
  // pair slots in the order of the pairs' first blocks
  if (t < W) {
    const bool low = partner_s[t] > t;
    const uint32_t bl = __ballot_sync(0xffffffffu, low);
    if (lane == 0) lower_s[t >> 5] = bl;
  }
  __syncthreads();
  if (t < W && partner_s[t] > t) {
    const uint64_t lowm = (uint64_t)(uint32_t)lower_s[0] | ((uint64_t)(uint32_t)lower_s[1] << 32);
    const int k = __popcll(lowm & ((1ull << t) - 1ull));
    prow[(int64_t)h * items + W / 2 * w + k] = (r0 + t) | ((r0 + partner_s[t]) << 16);
  }
}

// ------------------------------------------------------------------------------------
// Kept-block lists (CSR) from the best drop sets; special query rows keep everything.
// One warp per attention item: query rows 2u and 2u + 1 on the 64-token grid, row u on the
// 128-token grid.  With plist set the warp also writes the item's list for the attention
// kernel (what k_pairs builds from a caller's CSR): the union of its rows' lists, entry
// j | mask << 16 (bit 0: the item's first 64 query rows keep j, bit 1: the second 64), at the
// offset of the item's first row, and the union's length in plen.  Order: the blocks kept by
// one row only alternate between the rows first (see below), then the rest ascending.
// grid (ceil(items / 8), H) x 256 threads.
// ------------------------------------------------------------------------------------
struct CsrBases {
  int64_t base[RESS_MAX_HEADS + 1];
};

struct CsrOut {
  int32_t* row_ptr;
  int32_t* col_idx;
  int64_t cap;           // col_idx entries
  float* J_best;         // optional
  uint32_t* drop_mask;   // optional
  int32_t* plist;        // optional: attention item lists
  int32_t* plen;         // [H * items] with plist
  int64_t plist_cap;
  const int32_t* prow;   // optional: rows of items u < npaired (k_pairing), else adjacent
  int npaired;
  uint32_t* status;
  int rows_per_item;     // 2 on the 64-token grid, 1 on the 128-token grid
  bool variable;         // row offsets from row_ptr (k_rowptr) instead of the fixed budgets
};

// Row offsets of variable-length kept lists (CDF threshold): row_ptr = exclusive scan of the
// kept counts over the H * nq rows (candidate rows: kcount; special query rows: nb).  One
// CTA of 1024 threads, each owning a contiguous run of rows.
__global__ void __launch_bounds__(1024) k_rowptr(const int32_t* __restrict__ kcount, int H,
                                                 int nq, int nqc, int nb,
                                                 int32_t* __restrict__ row_ptr) {
  __shared__ long long wsum[32];
  const long long R = (long long)H * nq;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const long long per = (R + 1023) / 1024;
  const long long r0 = min(R, (long long)t * per), r1 = min(R, r0 + per);
  auto count = [&](long long r) -> long long { return (r % nq) >= nqc ? nb : kcount[r]; };
  long long local = 0;
  for (long long r = r0; r < r1; ++r) local += count(r);
  long long inc = local;  // inclusive scan over the warp, then over the warps
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long y = __shfl_up_sync(kFull, inc, o);
    if (lane >= o) inc += y;
  }
  if (lane == 31) wsum[warp] = inc;
  __syncthreads();
  if (warp == 0) {
    long long w = wsum[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(kFull, w, o);
      if (lane >= o) w += y;
    }
    wsum[lane] = w;
  }
  __syncthreads();
  long long off = inc - local + (warp ? wsum[warp - 1] : 0);
  for (long long r = r0; r < r1; ++r) {
    row_ptr[r] = (int32_t)off;
    off += count(r);
  }
  if (t == 1023) row_ptr[R] = (int32_t)off;
}

// The kept blocks of one mask word w of a row, written from list position `at` on.
__device__ __forceinline__ void csr_write_word(const CsrOut& o, uint32_t bits, int w, int at,
                                               int expect, int64_t off) {
  for (; bits; bits &= bits - 1u, ++at)
    if (at < expect && off + at < o.cap) o.col_idx[off + at] = w * 32 + (__ffs(bits) - 1);
}

__global__ void k_csr(SelPtrs p, Budgets bud, CsrBases cb, int H, CsrOut o) {
  const int h = blockIdx.y, lane = threadIdx.x & 31;
  const int rpi = o.rows_per_item;
  const int items = (p.nq + rpi - 1) / rpi;
  const int u = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (u >= items) return;
  const int i0 = u * rpi;
  const bool paired = o.prow && u < o.npaired;
  const int32_t pr = paired ? o.prow[(int64_t)h * items + u] : 0;
  const int rowi[2] = {paired ? (pr & 0xffff) : i0, paired ? (pr >> 16) : i0 + 1};
  const int nr = paired ? 2 : min(rpi, p.nq - i0);  // rows of this item: 1 or 2
  const int ns = p.nb - p.ncand;        // always-kept key blocks
  const int c = bud.c[h];
  int64_t ri[2], off[2];
  int expect[2], pos[2] = {0, 0};
  bool dense[2];
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int i = min(rowi[r], p.nq - 1);
    ri[r] = (int64_t)h * p.nq + i;
    dense[r] = i >= p.nqc;
    // fixed budgets: offsets by formula; variable lengths: the offsets k_rowptr wrote
    off[r] = o.variable ? (int64_t)o.row_ptr[ri[r]]
                        : cb.base[h] + (dense[r] ? (int64_t)p.nqc * (c + ns) +
                                                       (int64_t)(i - p.nqc) * p.nb
                                                 : (int64_t)i * (c + ns));
    expect[r] = o.variable ? (int)(o.row_ptr[ri[r] + 1] - off[r]) : (dense[r] ? p.nb : c + ns);
  }
  // an item's union list goes to its slot, the CSR span of rows rpi u .. rpi u + rpi - 1;
  // a paired item's two candidate rows have the slot's two lengths (fixed budgets)
  const int64_t uoff = paired ? cb.base[h] + (int64_t)i0 * (c + ns) : off[0];
  // best drop set of row r in mask word w (none for a dense row), and its kept blocks
  auto drop_word = [&](int r, int w) -> uint32_t {
    return dense[r] ? 0u : p.bmask[ri[r] * p.words + w];
  };
  auto kept_word = [&](int r, int w) -> uint32_t { return ~drop_word(r, w) & valid_bits(w, p.nb); };
  // Union list order: the k-th block kept by the first row only and the k-th kept by the
  // second only (k < P, the smaller of the two counts, both ascending) alternate at
  // positions 2k, 2k + 1, so that in the attention the two halves' softmax work of
  // consecutive one-sided tiles overlaps; then the rest of the union in ascending order.
  int P = 0;
  if (o.plist && rpi == 2 && nr == 2) {
    int nA = 0, nB = 0;
    for (int w = lane; w < p.words; w += 32) {
      const uint32_t ka = kept_word(0, w), kb = kept_word(1, w);
      nA += __popc(ka & ~kb);
      nB += __popc(kb & ~ka);
    }
    P = min(__reduce_add_sync(kFull, nA), __reduce_add_sync(kFull, nB));
  }
  // Lane l owns word w0 + l of each row: warp scans of the lanes' counts give every word's
  // first list positions, then each lane writes the blocks of its own word.
  int posU = 0, cA = 0, cB = 0, cR = 0;
  for (int w0 = 0; w0 < p.words; w0 += 32) {
    const int w = w0 + lane;
    uint32_t keep[2] = {0u, 0u};
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      if (r < nr && w < p.words) {
        const uint32_t dm = drop_word(r, w);
        if (o.drop_mask) o.drop_mask[ri[r] * p.words + w] = dm;
        keep[r] = ~dm & valid_bits(w, p.nb);
      }
    }
    // a 128-token query block keeps its list for both 64-row halves of the tile
    const uint32_t kb = rpi == 1 ? keep[0] : keep[1];
    const uint32_t un = o.plist ? (keep[0] | kb) : 0u;
    const uint32_t oa = P ? keep[0] & ~kb : 0u, ob = P ? kb & ~keep[0] : 0u;  // one-sided
    const int cAB = __popc(keep[0]) | (__popc(keep[1]) << 16), cU = __popc(un);
    const int cO = __popc(oa) | (__popc(ob) << 16);
    int iAB = cAB, iU = cU, iO = cO;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int yAB = __shfl_up_sync(kFull, iAB, d), yU = __shfl_up_sync(kFull, iU, d);
      const int yO = __shfl_up_sync(kFull, iO, d);
      if (lane >= d) {
        iAB += yAB;
        iU += yU;
        iO += yO;
      }
    }
    const int tAB = __shfl_sync(kFull, iAB, 31), tU = __shfl_sync(kFull, iU, 31);
    const int tO = __shfl_sync(kFull, iO, 31);
    csr_write_word(o, keep[0], w, pos[0] + ((iAB - cAB) & 0xffff), expect[0], off[0]);
    csr_write_word(o, keep[1], w, pos[1] + ((iAB - cAB) >> 16), expect[1], off[1]);
    if (o.plist) {
      // ranks of this word's first one-sided blocks; its lowest mA (mB) of them alternate
      const int gA = cA + ((iO - cO) & 0xffff), gB = cB + ((iO - cO) >> 16);
      const int mA = min(max(P - gA, 0), __popc(oa)), mB = min(max(P - gB, 0), __popc(ob));
      const int cRest = cU - mA - mB;
      int iR = cRest;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int y = __shfl_up_sync(kFull, iR, d);
        if (lane >= d) iR += y;
      }
      int kA = 0, kB = 0, at = 2 * P + cR + iR - cRest;
      for (uint32_t bits = un; bits; bits &= bits - 1u) {
        const int b = __ffs(bits) - 1;
        const int j = w * 32 + b;
        int64_t dst;
        int e;
        if ((oa >> b) & 1u) {
          dst = kA < mA ? 2 * (gA + kA) : at++;
          e = j | (1 << 16);
          ++kA;
        } else if ((ob >> b) & 1u) {
          dst = kB < mB ? 2 * (gB + kB) + 1 : at++;
          e = j | (2 << 16);
          ++kB;
        } else {
          dst = at++;
          e = j | (((int)((keep[0] >> b) & 1u) | (int)(((kb >> b) & 1u) << 1)) << 16);
        }
        if (uoff + dst < o.plist_cap) o.plist[uoff + dst] = e;
      }
      cR += __shfl_sync(kFull, iR, 31);
    }
    pos[0] += tAB & 0xffff;
    pos[1] += tAB >> 16;
    posU += tU;
    cA += tO & 0xffff;
    cB += tO >> 16;
  }
  if (lane == 0) {
    for (int r = 0; r < nr; ++r) {
      if (pos[r] != expect[r]) flag_status(o.status, kStatusBadRow);
      if (!o.variable) o.row_ptr[ri[r]] = (int32_t)off[r];
      if (o.J_best) o.J_best[ri[r]] = dense[r] ? 0.f : p.Jbest[ri[r]];
    }
    if (!o.variable && h == H - 1 && u == items - 1) o.row_ptr[(int64_t)H * p.nq] = (int32_t)cb.base[H];
    if (o.plist) o.plen[(int64_t)h * items + u] = posU;
  }
}

// ------------------------------------------------------------------------------------
// Failure detection without a fault: one thread waits on a shared-memory barrier that
// nothing arrives at, with the bounded wait of the kernels (a time limit, here also an
// iteration limit), and records the timeout in the status word as a kernel's wait does.
// ------------------------------------------------------------------------------------
__global__ void k_wait_selftest(uint32_t* status, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar, 1);
    ptx::fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    bool done = false;
    const uint64_t t0 = ptx::globaltimer();
    for (uint32_t it = 0; it < (1u << 24); ++it) {
      if (ptx::mbar_try_wait(&bar, 0)) {
        done = true;
        break;
      }
      if (ptx::globaltimer() - t0 > limit_ns) break;
    }
    if (!done) flag_status(status, kStatusTimeout);
  }
}

cudaError_t launch_wait_selftest(uint32_t* status, uint64_t limit_ns, cudaStream_t st) {
  k_wait_selftest<<<1, 32, 0, st>>>(status, limit_ns);
  note_launch();
  return cudaGetLastError();
}

// ------------------------------------------------------------------------------------
// launchers
// ------------------------------------------------------------------------------------

cudaError_t launch_prepare_wo(const Shape& s, const uint16_t* W_o, float* F, cudaStream_t st) {
  k_prepare_wo<<<s.H, kThreads, 0, st>>>(W_o, s.d_model, s.H, F);
  note_launch();
  return cudaGetLastError();
}

static Budgets budgets_of(const SelectArgs& a) {
  Budgets b;
  for (int h = 0; h < RESS_MAX_HEADS; ++h) b.c[h] = a.c[h];
  return b;
}

cudaError_t launch_score(const SelectArgs& a, cudaStream_t st) {
  const Shape& s = a.s;
  SelPtrs p = sel_ptrs(s, a.ws, a.L);
  float* qbar = (float*)(a.ws + a.L.qbar);
  float* kbar = (float*)(a.ws + a.L.kbar);
  float* vbar = (float*)(a.ws + a.L.vbar);
  float* ztil = (float*)(a.ws + a.L.ztil);
  k_pool<<<dim3(s.nb, 3), kThreads, 0, st>>>(a.Q, a.K, a.V, s.N, s.H, s.nb, s.qb, s.nq, qbar,
                                              kbar, vbar,
                                              (uint16_t*)(a.ws + a.L.asplit),
                                              (uint16_t*)(a.ws + a.L.ksplit));
  note_launch();
  k_zproj<<<dim3((s.nb + 15) / 16, s.H), kThreads, 0, st>>>(
      a.F, vbar, s.nb, ztil, (uint16_t*)(a.ws + a.L.zsplit), (int64_t)s.H * s.nb * kHeadDim,
      (float*)(a.ws + a.L.nz));
  note_launch();
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || s.ncand <= 0 || s.nqc <= 0) return e;
  // pooled logits, then P and y~, then q (Sec. 4.1, Eq. 1, Eq. 9), on the tensor cores
  if ((e = launch_logits(a, st)) != cudaSuccess) return e;
  if ((e = launch_yagg(a, st)) != cudaSuccess) return e;
  if ((e = launch_drift_norms(a, st)) != cudaSuccess) return e;
  const size_t rsmem =
      (size_t)kRowWarps * warp_scratch_words(s.ld, score_mask_words(s.words, a.v.cdf > 0.f)) * 4;
  auto kern = a.v.key == 0 ? k_score_rows<0> : a.v.key == 1 ? k_score_rows<1> : k_score_rows<2>;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)rsmem);
  if (e != cudaSuccess) return e;
  kern<<<dim3((s.nqc + kRowWarps - 1) / kRowWarps, s.H), 32 * kRowWarps, rsmem, st>>>(
      p, budgets_of(a), a.v);
  note_launch();
  return cudaGetLastError();
}

cudaError_t launch_round(const SelectArgs& a, int round, float rho, cudaStream_t st) {
  const Shape& s = a.s;
  if (s.ncand <= 0 || s.nqc <= 0) return cudaSuccess;
  SelPtrs p = sel_ptrs(s, a.ws, a.L);
  cudaError_t e = launch_gain(a, round, rho, st);  // t_ij on the tensor cores
  if (e != cudaSuccess) return e;
  const size_t rsmem = (size_t)kRowWarps * warp_scratch_words(s.ld, 3 * s.words) * 4;
  auto kern = a.v.direction != 0 ? k_round_rows<1> : k_round_rows<0>;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)rsmem);
  if (e != cudaSuccess) return e;
  kern<<<dim3((s.nqc + kRowWarps - 1) / kRowWarps, s.H), 32 * kRowWarps, rsmem, st>>>(
      p, budgets_of(a), round, rho);
  note_launch();
  return cudaGetLastError();
}

cudaError_t launch_csr(const SelectArgs& a, const int64_t* head_base, int32_t* row_ptr,
                       int32_t* col_idx, int64_t col_capacity, float* J_best,
                       uint32_t* drop_mask, int32_t* plist, int32_t* plen, int64_t plist_cap,
                       const int32_t* prow, cudaStream_t st) {
  const Shape& s = a.s;
  SelPtrs p = sel_ptrs(s, a.ws, a.L);
  CsrBases cb;
  for (int h = 0; h <= s.H; ++h) cb.base[h] = head_base[h];
  CsrOut o;
  o.row_ptr = row_ptr;
  o.col_idx = col_idx;
  o.cap = col_capacity;
  o.J_best = J_best;
  o.drop_mask = drop_mask;
  o.plist = plist;
  o.plen = plen;
  o.plist_cap = plist_cap;
  o.status = (uint32_t*)(a.ws + a.L.status);
  o.rows_per_item = s.qb == 128 ? 1 : 2;
  o.variable = a.v.cdf > 0.f;
  o.prow = prow;
  o.npaired = prow ? paired_items(s) : 0;
  if (o.variable) {
    k_rowptr<<<1, 1024, 0, st>>>(p.kcount, s.H, s.nq, s.nqc, s.nb, row_ptr);
    note_launch();
  }
  const int items = (s.nq + o.rows_per_item - 1) / o.rows_per_item;
  k_csr<<<dim3((items + 7) / 8, s.H), 256, 0, st>>>(p, budgets_of(a), cb, s.H, o);
  note_launch();
  return cudaGetLastError();
}

bool pairing_active(const Shape& s, const Variant& v) {
  return s.qb == kBlock && v.cdf <= 0.f && paired_items(s) > 0;
}

int paired_items(const Shape& s) { return s.nqc / 2; }

cudaError_t launch_pairing(const SelectArgs& a, int32_t* prow, cudaStream_t st) {
  const Shape& s = a.s;
  const int npaired = paired_items(s);
  const int windows = (2 * npaired + kPairWindow - 1) / kPairWindow;
  const size_t smem = (size_t)kPairWindow * ((((s.words + 1) >> 1) | 1) * 8);
  cudaError_t e = cudaFuncSetAttribute(k_pairing, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_pairing<<<dim3(windows, s.H), 512, smem, st>>>((const uint32_t*)(a.ws + a.L.bmask), s.nq, s.words,
                                                   s.ncand, npaired, (s.nb + 1) / 2, prow);
  note_launch();
  return cudaGetLastError();
}

}  // namespace ress
