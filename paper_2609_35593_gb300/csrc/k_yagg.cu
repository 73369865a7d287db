// Pooled attention map and pooled output in F space (Sec. 4.1, Eq. 1) on the tensor cores:
//   P_ij = 2^(L_ij - m_i) / Z_i   over all key blocks j < nb   (L = pooled logits in base-2
//                                                                 units, from k_dot)
//   y~_i = sum_j P_ij z~_j                                     (z~_j = F_h V_j)
// for the candidate rows of one head.  m_i and Z_i come from the per-slice maxima and sums
// k_dot left in lstat.  P overwrites L in place; y~ is written in fp32, as three bf16
// terms (the row operand of the drift-norm products) and as ||y~_i||^2.
//
// One CTA per 128 candidate rows of a head and part of the key blocks (the blocks are split
// into `parts` consecutive ranges of chunks when that fills more of the GPU; each part's
// partial y~ goes to scratch and the CTA that finishes last sums the parts in their order and
// writes the outputs, so the result does not depend on which finishes first), 544 threads,
// 64 key blocks per chunk, two pipeline stages:
//   warp 16    lane 0 loads chunk c + 1 by TMA (L: two 32-column fp32 boxes; z~: its three
//              bf16 term tiles, 64 blocks x 64 channels) while the chunk c is converted;
//              then the converged warp, one elected lane, issues the chunk's MMAs
//                y~ += P_c^(a) z~_c^(b)   for the six term pairs (a, b) of k_dot,
//              M128 N64 K16 x 4 each, P terms K-major, z~ terms MN-major, both from shared
//              memory, and commits them to the stage's "empty" barrier;
//   warps 0-15 one row and 16 of the chunk's blocks per thread: P from L, written back over
//              its logits in the stage buffer and as three bf16 terms into the stage's A
//              tiles (128-byte swizzle); once all converters have done so (a bounded
//              mbarrier), the chunk's 128 x 64 block of P goes to global memory as whole
//              256-byte row segments, then an arrive on the stage's "converted" barrier;
//              after the last chunk the epilogue (warp w: TMEM lanes 32 (w mod 4)..,
//              columns 16 (w / 4)..).
// Every mbarrier wait is bounded; a wait that gives up records RESS_ETIMEOUT, lets copies
// and MMAs already issued finish (again bounded), frees TMEM and returns.

#include <cudaTypedefs.h>

#include "ress_internal.cuh"
#include "sm100_ptx.cuh"

namespace ress {
using namespace ptx;

bool make_term_map(CUtensorMap* m, const void* base, int nb, int H, int rows);
bool make_row_map(CUtensorMap* m, void* base, int nb, int H, int ld);

namespace {

constexpr int kConvWarps = 16;
constexpr int kYThreads = 32 * kConvWarps + 32;
constexpr int kMmaWarp = kConvWarps;
constexpr int kYRows = 128;      // candidate rows per CTA
constexpr int kYChunk = 64;      // key blocks per pipeline step
constexpr int kYStages = 2;
constexpr uint32_t kYCols = 64;  // TMEM columns: y~ (128 x 64 fp32)
constexpr uint64_t kYWaitNs = 2000000000ull;
constexpr uint64_t kYDrainNs = 200000000ull;

struct __align__(1024) YSmem {
  uint8_t L[kYStages][2][16384];  // logits: 2 boxes of 128 rows x 32 fp32 (swizzled)
  uint8_t A[kYStages][3][16384];  // P terms: 128 rows x 64 blocks bf16 (K-major, swizzled)
  uint8_t Z[kYStages][3][8192];   // z~ terms: 64 blocks x 64 channels bf16 (MN-major)
  float ny_part[4][kYRows];
  uint64_t full[kYStages], conv[kYStages], empty[kYStages];
  uint64_t pdone[kYStages];  // every converter's P is in the stage's logits buffer
  uint64_t done;
  uint32_t tmem_base;
  int abort;
  int last;  // this CTA sums the parts
};

struct YParams {
  int nb, nq, nqc, ld, nslices, nchunks;  // key blocks, query blocks, candidate query blocks
  const float2* lstat;
  float* P;         // [H, nb, ld]: logits in, probabilities out
  float* ytil;      // [H, nb, 64]
  uint32_t* asplit; // bf16x2 [3][H][nb][32]
  float* ny;        // [H, nb]
  int64_t term_words;  // H nb 32
  uint32_t* status;
  int parts;           // key-block parts per stripe of 128 rows
  float* part_buf;     // [parts][H][nq][64] partial y~ (parts > 1)
  uint32_t* arrivals;  // [H][stripes] parts done, zero before the launch (parts > 1)
};

// (A term, B term) of product q of the six, smallest first (as in k_dot).
constexpr uint32_t kTermA = 0x010201u;
constexpr uint32_t kTermB = 0x001021u;

__device__ __forceinline__ bool y_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort, kYWaitNs) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

// Barrier among the converter warps only (named barrier 1; the MMA warp takes no part).
__device__ __forceinline__ void conv_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(32 * kConvWarps) : "memory");
}

__device__ __forceinline__ void y_give_up(YSmem& S, uint32_t* status) {
  flag_status(status, kStatusTimeout);
  *reinterpret_cast<volatile int*>(&S.abort) = 1;
}

__global__ void __launch_bounds__(kYThreads, 1)
    k_yagg(const __grid_constant__ CUtensorMap tmL, const __grid_constant__ CUtensorMap tmZ,
           const YParams p) {
  extern __shared__ uint8_t smem_raw[];
  YSmem& S = *reinterpret_cast<YSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                       ~static_cast<uintptr_t>(1023));
  const int h = blockIdx.y, i0 = blockIdx.x * kYRows, part = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &S.abort;
  // this part's chunks [c0, c1); the pipeline counts them from 0
  const int c0 = (int)((int64_t)p.nchunks * part / p.parts);
  const int nch = (int)((int64_t)p.nchunks * (part + 1) / p.parts) - c0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kYStages; ++s) {
      mbar_init(&S.full[s], 1);
      mbar_init(&S.conv[s], kConvWarps);
      mbar_init(&S.pdone[s], kConvWarps);
      mbar_init(&S.empty[s], 1);
    }
    mbar_init(&S.done, 1);
    S.abort = 0;
    fence_barrier_init();
    prefetch_tensormap(&tmL);
    prefetch_tensormap(&tmZ);
  }
  if (warp == kMmaWarp) tmem_alloc(&S.tmem_base, kYCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = S.tmem_base;

  if (warp == kMmaWarp) {
    // ============================ loads and MMAs ====================================
    const bool leader = elect_one();
    bool failed = false;
    if (__popc(__ballot_sync(0xffffffffu, leader)) != 1) {
      if (lane == 0) flag_status(p.status, kStatusBadRow);
      *abort = 1;
      failed = true;
    }
    int produced = 0, consumed = 0;
    auto produce = [&](int c) -> bool {
      const int s = c % kYStages, u = c / kYStages;
      if (u > 0 && !y_wait(&S.empty[s], (u - 1) & 1, abort)) return false;
      if (lane == 0) {
        const int j0 = (c0 + c) * kYChunk;
        mbar_arrive_expect_tx(&S.full[s], 2 * 16384 + 3 * 8192);
        tma_load_3d(S.L[s][0], &tmL, &S.full[s], j0, i0, h);
        tma_load_3d(S.L[s][1], &tmL, &S.full[s], j0 + 32, i0, h);
#pragma unroll
        for (int t = 0; t < 3; ++t) tma_load_4d(S.Z[s][t], &tmZ, &S.full[s], 0, j0, h, t);
      }
      __syncwarp();
      ++produced;
      return true;
    };
    const uint32_t idesc = idesc_bf16_f32(kYRows, 64, true);
    if (!failed && !produce(0)) failed = true;
    for (int c = 0; c < nch && !failed; ++c) {
      if (c + 1 < nch && !produce(c + 1)) {
        failed = true;
        break;
      }
      const int s = c % kYStages, par = (c / kYStages) & 1;
      if (!y_wait(&S.full[s], par, abort) || !y_wait(&S.conv[s], par, abort)) {
        failed = true;
        break;
      }
      tc_fence_after();
      if (leader) {
#pragma unroll
        for (int q = 0; q < 6; ++q) {
          const uint32_t a = smem_u32(S.A[s][(kTermA >> (4 * q)) & 0xF]);
          const uint32_t b = smem_u32(S.Z[s][(kTermB >> (4 * q)) & 0xF]);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            mma_bf16_ss(tmem, sdesc_sw128(a + 32 * k), sdesc_sw128(b + 2048 * k), idesc,
                        (c > 0 || q > 0 || k > 0) ? 1u : 0u);
        }
        mma_commit(&S.empty[s]);
        if (c + 1 == nch) mma_commit(&S.done);
      }
      __syncwarp();
      ++consumed;
    }
    if (failed) {
      if (lane == 0) {
        y_give_up(S, p.status);
        volatile int no_abort = 0;
        // copies issued and MMAs committed must finish before the memory goes away
        for (int c = consumed; c < produced; ++c)
          mbar_wait(&S.full[c % kYStages], (c / kYStages) & 1, &no_abort, kYDrainNs);
        if (consumed > 0) {
          const int c = consumed - 1;
          mbar_wait(&S.empty[c % kYStages], (c / kYStages) & 1, &no_abort, kYDrainNs);
        }
      }
      __syncwarp();
    }
  } else {
    // ============================ conversion ========================================
    const int r = 32 * (warp & 3) + lane, qq = warp >> 2;  // row of the tile, column quarter
    const int i = i0 + r;
    const bool row_ok = i < p.nqc;
    const int64_t ri = (int64_t)h * p.nq + i;
    float m = 0.f, iz = 0.f;
    if (row_ok) {  // the row's softmax from its per-slice maxima and sums
      m = -INFINITY;
      for (int t = 0; t < p.nslices; ++t) m = fmaxf(m, p.lstat[ri * p.nslices + t].x);
      float z = 0.f;
      for (int t = 0; t < p.nslices; ++t) {
        const float2 st = p.lstat[ri * p.nslices + t];
        if (st.x != -INFINITY) z += st.y * exp2f(st.x - m);
      }
      iz = 1.0f / z;
    }
    bool failed = false;
    for (int c = 0; c < nch; ++c) {
      const int s = c % kYStages, par = (c / kYStages) & 1;
      if (!y_wait(&S.full[s], par, abort)) {
        failed = true;
        break;
      }
      const int jb = (c0 + c) * kYChunk + 16 * qq;  // first block of this thread's 16
      // L: box qq / 2, 16-byte chunks 4 (qq mod 2) .. + 3 of row r
      uint8_t* lrow = S.L[s][qq >> 1] + r * 128;
      float pv[16];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float4 v = *reinterpret_cast<const float4*>(lrow + (((4 * (qq & 1) + k) ^ (r & 7)) << 4));
        const float lv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e)
          pv[4 * k + e] = (row_ok && jb + 4 * k + e < p.nb) ? ex2(lv[e] - m) * iz : 0.f;
      }
      // P back over this thread's logits in the stage buffer and its three bf16 terms into
      // the A tiles; once every converter has done so, the chunk's 128 x 64 block of P goes
      // to global memory as whole row segments (two 256-byte rows per warp and store
      // instead of 32 rows of 16 bytes)
#pragma unroll
      for (int k = 0; k < 4; ++k)
        *reinterpret_cast<float4*>(lrow + (((4 * (qq & 1) + k) ^ (r & 7)) << 4)) =
            make_float4(pv[4 * k], pv[4 * k + 1], pv[4 * k + 2], pv[4 * k + 3]);
      // P terms: this thread's 16 blocks are 16-byte chunks 2 qq, 2 qq + 1 of row r
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        uint32_t hi[4], mid[4], lo[4];
#pragma unroll
        for (int e = 0; e < 4; ++e)
          split3_bf16x2(pv[8 * k + 2 * e], pv[8 * k + 2 * e + 1], hi[e], mid[e], lo[e]);
        const int off = r * 128 + (((2 * qq + k) ^ (r & 7)) << 4);
        *reinterpret_cast<uint4*>(S.A[s][0] + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        *reinterpret_cast<uint4*>(S.A[s][1] + off) = make_uint4(mid[0], mid[1], mid[2], mid[3]);
        *reinterpret_cast<uint4*>(S.A[s][2] + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&S.pdone[s]);
      if (!y_wait(&S.pdone[s], par, abort)) {  // bounded: a converter that gave up ends it
        failed = true;
        break;
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int idx = (int)threadIdx.x + 32 * kConvWarps * k;  // float4 of the 128 x 16
        const int rr = idx >> 4, c4 = idx & 15;
        const int j = (c0 + c) * kYChunk + 4 * c4;
        if (i0 + rr < p.nqc && j < p.ld) {  // ld is a multiple of 16
          const float4 v4 = *reinterpret_cast<const float4*>(
              S.L[s][c4 >> 3] + rr * 128 + (((c4 & 7) ^ (rr & 7)) << 4));
          *reinterpret_cast<float4*>(p.P + ((int64_t)h * p.nq + i0 + rr) * p.ld + j) = v4;
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&S.conv[s]);
    }
    if (failed && lane == 0) y_give_up(S, p.status);
    // ---- epilogue: y~ row r, channels 16 qq .. 16 qq + 15 ------------------------------
    float nyp = 0.f;
    bool have = false;
    uint32_t v[16];
    if (!failed && y_wait(&S.done, 0, abort)) {
      tc_fence_after();
      RESS_TMEM_LD16(tmem + ((uint32_t)(32 * (warp & 3)) << 16) + 16 * qq, v);
      have = true;
    } else if (lane == 0) {
      y_give_up(S, p.status);
    }
    if (p.parts > 1) {
      // this part's sums to scratch; the last part to arrive adds all parts in order
      float* mine = p.part_buf + (((int64_t)part * gridDim.y + h) * p.nq + (row_ok ? i : 0)) * 64 + 16 * qq;
      if (have && row_ok) {
#pragma unroll
        for (int k = 0; k < 4; ++k)
          *reinterpret_cast<float4*>(mine + 4 * k) =
              make_float4(__uint_as_float(v[4 * k]), __uint_as_float(v[4 * k + 1]),
                          __uint_as_float(v[4 * k + 2]), __uint_as_float(v[4 * k + 3]));
      }
      __threadfence();
      conv_sync();
      if (threadIdx.x == 0) {
        const uint32_t before = atomicAdd(&p.arrivals[h * gridDim.x + blockIdx.x], 1u);
        S.last = before == (uint32_t)(p.parts - 1);
        if (S.last) p.arrivals[h * gridDim.x + blockIdx.x] = 0u;  // ready for the next call
      }
      conv_sync();
      have = have && S.last;
      if (have && row_ok) {
        __threadfence();
        float acc[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) acc[k] = 0.f;
        for (int t = 0; t < p.parts; ++t) {
          const float* src = p.part_buf + (((int64_t)t * gridDim.y + h) * p.nq + i) * 64 + 16 * qq;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float4 q4 = __ldcg(reinterpret_cast<const float4*>(src + 4 * k));
            acc[4 * k] += q4.x;
            acc[4 * k + 1] += q4.y;
            acc[4 * k + 2] += q4.z;
            acc[4 * k + 3] += q4.w;
          }
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = __float_as_uint(acc[k]);
      }
    }
    if (have) {
      if (row_ok) {
        float* yrow = p.ytil + ri * 64 + 16 * qq;
#pragma unroll
        for (int k = 0; k < 4; ++k)
          *reinterpret_cast<float4*>(yrow + 4 * k) =
              make_float4(__uint_as_float(v[4 * k]), __uint_as_float(v[4 * k + 1]),
                          __uint_as_float(v[4 * k + 2]), __uint_as_float(v[4 * k + 3]));
        uint32_t* as = p.asplit + ri * 32 + 8 * qq;
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          uint32_t hi[4], mid[4], lo[4];
#pragma unroll
          for (int e = 0; e < 4; ++e)
            split3_bf16x2(__uint_as_float(v[8 * k + 2 * e]), __uint_as_float(v[8 * k + 2 * e + 1]),
                          hi[e], mid[e], lo[e]);
          *reinterpret_cast<uint4*>(as + 4 * k) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
          *reinterpret_cast<uint4*>(as + p.term_words + 4 * k) =
              make_uint4(mid[0], mid[1], mid[2], mid[3]);
          *reinterpret_cast<uint4*>(as + 2 * p.term_words + 4 * k) =
              make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) nyp = fmaf(__uint_as_float(v[k]), __uint_as_float(v[k]), nyp);
      }
    }
    S.ny_part[qq][r] = nyp;
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < kYRows && (p.parts == 1 || S.last)) {
    const int i = i0 + threadIdx.x;
    if (i < p.nqc && !*abort)
      p.ny[(int64_t)h * p.nq + i] = (S.ny_part[0][threadIdx.x] + S.ny_part[1][threadIdx.x]) +
                                    (S.ny_part[2][threadIdx.x] + S.ny_part[3][threadIdx.x]);
  }
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kYCols);
  }
}

}  // namespace

cudaError_t launch_yagg(const SelectArgs& a, cudaStream_t st) {
  const Shape& s = a.s;
  if (s.ncand <= 0 || s.nqc <= 0) return cudaSuccess;
  CUtensorMap tl, tz;
  if (!make_row_map(&tl, a.ws + a.L.P, s.nq, s.H, s.ld) ||
      !make_term_map(&tz, a.ws + a.L.zsplit, s.nb, s.H, kYChunk))
    return cudaErrorInvalidValue;
  YParams p;
  p.nb = s.nb;
  p.nq = s.nq;
  p.nqc = s.nqc;
  p.ld = s.ld;
  p.nslices = (s.nb + 127) / 128;
  p.nchunks = (s.nb + kYChunk - 1) / kYChunk;
  p.lstat = (const float2*)(a.ws + a.L.lstat);
  p.P = (float*)(a.ws + a.L.P);
  p.ytil = (float*)(a.ws + a.L.ytil);
  p.asplit = (uint32_t*)(a.ws + a.L.asplit);
  p.ny = (float*)(a.ws + a.L.ny);
  p.term_words = (int64_t)s.H * s.nq * 32;
  p.status = (uint32_t*)(a.ws + a.L.status);
  // One CTA per SM: when the stripes of rows leave SMs idle, split the key blocks into as
  // many parts (up to 3) as still run in one wave.  (A second wave costs more than the
  // split saves: measured at 32 views on 64-token query blocks, 96 stripes.)
  const int stripes = (s.nqc + kYRows - 1) / kYRows;
  int dev = 0, sms = 1;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  p.parts = 1;
  // (the partial sums of k parts take 64 k of the ld floats per row of the gains array)
  for (int k = 2; k <= 3 && k <= p.nchunks && 64 * k <= s.ld; ++k)
    if ((int64_t)stripes * s.H * k <= sms) p.parts = k;
  // scratch while the selection scores: the gains array (partial y~) and the attention
  // items' length array (arrival counts), both unused until the restoration rounds
  p.part_buf = (float*)(a.ws + a.L.t);
  p.arrivals = (uint32_t*)(a.ws + a.L.plen);
  cudaError_t e;
  if (p.parts > 1 &&
      (e = cudaMemsetAsync(p.arrivals, 0, (size_t)stripes * s.H * sizeof(uint32_t), st)) != cudaSuccess)
    return e;
  const size_t smem = sizeof(YSmem) + 1024;
  e = cudaFuncSetAttribute(k_yagg, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_yagg<<<dim3(stripes, s.H, p.parts), kYThreads, smem, st>>>(tl, tz, p);
  note_launch();
  return cudaGetLastError();
}

}  // namespace ress
