// Internal definitions shared by the ReSS CUDA translation units (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "../../include/ress.h"

namespace ress {

constexpr int kHeadDim = RESS_HEAD_DIM;  // d_h
constexpr int kBlock = RESS_BLOCK;       // 64x64 block grid
constexpr float kEps = 1e-4f;            // Eq. 7

// Device status word values (first error wins; read back by ress_status).
constexpr uint32_t kStatusTimeout = 1;
constexpr uint32_t kStatusBadIndex = 2;
constexpr uint32_t kStatusBadRow = 3;

// Derived sizes of one layer.
// Key blocks are 64 tokens (columns of the selection); query blocks qb = 64 or 128 tokens
// (rows of the selection, the CSR and the attention items).
struct Shape {
  int N, H, nb, ncand, nspecial_blocks, words, ld, d_model;
  int qb, nq, nqc;  // query block size, query blocks, candidate (sparsified) query blocks
};

inline Shape make_shape(const ress_dims& d) {
  Shape s;
  s.N = d.n_tokens;
  s.H = d.n_heads;
  s.nb = (d.n_tokens + kBlock - 1) / kBlock;
  s.ncand = (d.n_tokens - d.n_special) / kBlock;
  s.nspecial_blocks = s.nb - s.ncand;
  s.words = (s.nb + 31) / 32;
  s.ld = (s.nb + 31) / 32 * 32;
  s.d_model = d.d_model;
  s.qb = d.q_block == 128 ? 128 : kBlock;
  s.nq = (d.n_tokens + s.qb - 1) / s.qb;
  s.nqc = (d.n_tokens - d.n_special) / s.qb;
  return s;
}

inline int64_t align256(int64_t x) { return (x + 255) / 256 * 256; }

inline ress_ws_layout make_layout(const Shape& s) {
  ress_ws_layout L;
  int64_t off = 0;
  auto take = [&](int64_t bytes) {
    int64_t o = off;
    off = align256(off + bytes);
    return o;
  };
  const int64_t vec = (int64_t)s.H * s.nb * kHeadDim * 4;   // per key block
  const int64_t qvec = (int64_t)s.H * s.nq * kHeadDim * 4;  // per query block
  const int64_t mat = (int64_t)s.H * s.nq * s.ld * 4;
  const int64_t row = (int64_t)s.H * s.nq * 4;
  const int64_t msk = (int64_t)s.H * s.nq * s.words * 4;
  L.status = take(64);
  L.counter = take(64);
  L.qbar = take(qvec);
  L.kbar = take(vec);
  L.vbar = take(vec);
  L.ztil = take(vec);
  L.ytil = take(qvec);
  L.gtil = take(qvec);
  L.P = take(mat);
  L.q = take(mat);
  L.t = take(mat);
  L.K = take(row);
  L.G = take(row);
  L.J = take(row);
  L.Jbest = take(row);
  L.J0 = take(row);
  L.dmask = take(msk);
  L.bmask = take(msk);
  L.plen = take((int64_t)s.H * ((s.nb + 1) / 2) * 4);
  L.asplit = take(3 * (int64_t)s.H * s.nq * kHeadDim * 2);
  L.ksplit = take(3 * (int64_t)s.H * s.nb * kHeadDim * 2);
  L.zsplit = take(3 * (int64_t)s.H * s.nb * kHeadDim * 2);
  L.cdot = take(row);
  L.ny = take(row);
  L.nz = take((int64_t)s.H * s.nb * 4);
  L.lstat = take((int64_t)s.H * s.nq * ((s.nb + 127) / 128) * 8);
  L.kcount = take(row);
  L.prow = take((int64_t)s.H * ((s.nb + 1) / 2) * 4);
  L.ld = s.ld;
  L.words = s.words;
  L.total = off;
  return L;
}

// Record the first device-side failure in the workspace status word.
__device__ __forceinline__ void flag_status(uint32_t* status, uint32_t code) {
  atomicCAS(status, 0u, code);
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// Per-head kept-block budgets c_h (Eq. 7), passed to kernels by value.
struct Budgets {
  int c[RESS_MAX_HEADS];
};

// Swap count of round r (Eq. 17): floor(rho c_h / 2^(r+1)), capped by |D| and |P \ D|.
__host__ __device__ inline int swap_count(int c, int ncand, int round, float rho) {
  const int m = (int)floor((double)rho * (double)c / (double)(1ull << (round + 1)));
  return min(m, min(ncand - c, c));
}

// Two floats as sums of three bf16 terms each, every term rounded to nearest:
// x = hi + mid + lo up to |x| 2^-24 or so (hi carries the top 8 significant bits, mid
// the next 8, lo the rest; both subtractions are exact).  Packed bf16x2, x0 in the low half.
__device__ __forceinline__ uint32_t cvt_bf16x2(float lo_elem, float hi_elem) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi_elem), "f"(lo_elem));
  return r;
}
__device__ __forceinline__ uint16_t cvt_bf16(float x) {
  uint16_t r;
  asm("cvt.rn.bf16.f32 %0, %1;" : "=h"(r) : "f"(x));
  return r;
}
// One float as three bf16 terms (same rule as split3_bf16x2).
__device__ __forceinline__ void split3_bf16(float x, uint16_t& hi, uint16_t& mid, uint16_t& lo) {
  hi = cvt_bf16(x);
  const float r = x - __uint_as_float((uint32_t)hi << 16);
  mid = cvt_bf16(r);
  lo = cvt_bf16(r - __uint_as_float((uint32_t)mid << 16));
}
__device__ __forceinline__ void split3_bf16x2(float x0, float x1, uint32_t& hi, uint32_t& mid,
                                              uint32_t& lo) {
  hi = cvt_bf16x2(x0, x1);
  const float r0 = x0 - __uint_as_float(hi << 16), r1 = x1 - __uint_as_float(hi & 0xffff0000u);
  mid = cvt_bf16x2(r0, r1);
  const float s0 = r0 - __uint_as_float(mid << 16), s1 = r1 - __uint_as_float(mid & 0xffff0000u);
  lo = cvt_bf16x2(s0, s1);
}

// Streaming 16-byte load that bypasses L1 allocation (read-once inputs).
__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// Counts one kernel launch of this library (host side, process-wide; ress_kernel_launches).
void note_launch();

// Kernel launchers (defined in k_select.cu / k_attn.cu); each returns a cudaError_t.
// Selection variant (ress_variant) as the kernels take it.
struct Variant {
  int key;        // 0 drift (Eq. 7), 1 pooled probability, 2 random
  int direction;  // 0 minimise J, 1 restoration maximises J, 2 initial selection too
  unsigned long long seed;
  float cdf;      // 0 off; tau: keep further candidates until the kept mass reaches tau
};

struct SelectArgs {
  Shape s;
  const uint16_t *Q, *K, *V;
  const float* F;
  char* ws;
  ress_ws_layout L;
  int c[RESS_MAX_HEADS];
  Variant v;
};

cudaError_t launch_prepare_wo(const Shape& s, const uint16_t* W_o, float* F, cudaStream_t st);
cudaError_t launch_score(const SelectArgs& a, cudaStream_t st);
cudaError_t launch_round(const SelectArgs& a, int round, float rho, cudaStream_t st);
cudaError_t launch_gain(const SelectArgs& a, int round, float rho, cudaStream_t st);
cudaError_t launch_logits(const SelectArgs& a, cudaStream_t st);
cudaError_t launch_drift_norms(const SelectArgs& a, cudaStream_t st);
cudaError_t launch_yagg(const SelectArgs& a, cudaStream_t st);
// Kept-block lists in CSR form; with plist set, also the attention items' union lists and
// their lengths (what launch_attn_pairs builds from a caller's CSR), so that a forward can
// go straight to launch_attn_range.
cudaError_t launch_csr(const SelectArgs& a, const int64_t* head_base, int32_t* row_ptr,
                       int32_t* col_idx, int64_t col_capacity, float* J_best,
                       uint32_t* drop_mask, int32_t* plist, int32_t* plen, int64_t plist_cap,
                       const int32_t* prow, cudaStream_t st);
// Attention items of a forward on the 64-token grid with fixed budgets: the candidate query
// blocks are paired by the overlap of their best kept lists, within windows of
// kPairWindow blocks (prow, see ress_ws_layout); items of the window hold pair indices
// [kPairWindow/2 * w, ...).  pairing_active says whether a forward on this shape and
// variant uses the table; paired_items is the number of table entries per head.
constexpr int kPairWindow = 64;
bool pairing_active(const Shape& s, const Variant& v);
int paired_items(const Shape& s);
cudaError_t launch_pairing(const SelectArgs& a, int32_t* prow, cudaStream_t st);

struct AttnArgs {
  Shape s;
  const uint16_t *Q, *K, *V;
  const int32_t *row_ptr, *col_idx;
  int64_t col_capacity;
  void* O;              // bf16, or float32 when out_f32
  bool out_f32;
  uint32_t* status;
  uint32_t* counter;
  int32_t* plist;       // scratch: union lists of query-block pairs (>= scratch_cap entries)
  int32_t* plen;        // scratch: [H * ceil(nb / 2)] union lengths
  int64_t scratch_cap;
  const int32_t* prow;  // item table of a paired forward (items p < npaired), or NULL
  int npaired;
};
cudaError_t launch_sparse_attn(const AttnArgs& a, cudaStream_t st);
// The two halves of launch_sparse_attn, for callers that split the attention: the union
// lists of the query-block pairs, then the attention over pairs [p0, p1) of every head
// (query tokens [128 p0, 128 p1)) with tile-scheduler counter `slot`, which the caller
// zeroes before the launch.  Pairs are 128 query rows: two 64-token query blocks, or one
// 128-token block on the paper's grid.
constexpr int kAttnCounterSlots = 16;  // uint32 counters in the workspace's 64-byte slot
int attn_num_pairs(const Shape& s);
cudaError_t launch_attn_pairs(const AttnArgs& a, cudaStream_t st);
cudaError_t launch_attn_range(const AttnArgs& a, int p0, int p1, int slot, cudaStream_t st);

struct OProjArgs {
  int N, H, Dm;                      // tokens, heads (K = 64 H), d_model
  const uint16_t *O, *O2, *W_o, *x;  // O2: the second output (token drift)
  uint16_t* y;
  float* drift;
  uint32_t* status;
};
cudaError_t launch_out_proj(const OProjArgs& a, cudaStream_t st);
cudaError_t launch_token_drift(const OProjArgs& a, cudaStream_t st);

}  // namespace ress
