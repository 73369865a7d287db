// C ABI of the ReSS hot path: host-side validation, workspace layout and launch order.
// Every check happens before the first launch; nothing here allocates device memory.

#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <atomic>
#include <mutex>

#include "ress_internal.cuh"

namespace {

std::atomic<uint64_t> g_kernel_launches{0};

thread_local char g_err[512] = "";

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

int ok() {
  g_err[0] = '\0';
  return RESS_OK;
}

int check_dims(const ress_dims* d) {
  if (!d) return fail(RESS_EINVAL, "dims is NULL");
  if (d->head_dim != RESS_HEAD_DIM)
    return fail(RESS_EUNSUPPORTED, "head_dim %d unsupported (must be 64)", d->head_dim);
  if (d->block != RESS_BLOCK) return fail(RESS_EUNSUPPORTED, "block %d unsupported (must be 64)", d->block);
  if (d->n_heads < 1 || d->n_heads > RESS_MAX_HEADS)
    return fail(RESS_EUNSUPPORTED, "n_heads %d outside 1..%d", d->n_heads, RESS_MAX_HEADS);
  if (d->n_tokens < 1) return fail(RESS_EINVAL, "n_tokens %d < 1", d->n_tokens);
  if (d->n_special < 0 || d->n_special >= d->n_tokens)
    return fail(RESS_EINVAL, "n_special %d outside 0..n_tokens-1", d->n_special);
  if (d->d_model < 1) return fail(RESS_EINVAL, "d_model %d < 1", d->d_model);
  if (d->q_block != 0 && d->q_block != 64 && d->q_block != 128)
    return fail(RESS_EUNSUPPORTED, "q_block %d unsupported (0, 64 or 128)", d->q_block);
  const int64_t nb = ((int64_t)d->n_tokens + RESS_BLOCK - 1) / RESS_BLOCK;
  if (nb > RESS_MAX_BLOCKS)
    return fail(RESS_EUNSUPPORTED, "%lld blocks exceed the limit of %d", (long long)nb, RESS_MAX_BLOCKS);
  return RESS_OK;
}

int check_ptr(const void* p, size_t align, const char* name) {
  if (!p) return fail(RESS_EINVAL, "%s is NULL", name);
  if (reinterpret_cast<uintptr_t>(p) % align)
    return fail(RESS_EINVAL, "%s is not %zu-byte aligned", name, align);
  return RESS_OK;
}

int check_budgets(const ress::Shape& s, const int32_t* c) {
  if (!c) return fail(RESS_EINVAL, "c_h_host is NULL");
  for (int h = 0; h < s.H; ++h) {
    if (s.ncand > 0 && (c[h] < 1 || c[h] > s.ncand))
      return fail(RESS_EINVAL, "c_h[%d] = %d outside 1..|P| = %d", h, c[h], s.ncand);
    if (s.ncand == 0 && c[h] != 0)
      return fail(RESS_EINVAL, "c_h[%d] = %d but there are no candidate blocks", h, c[h]);
  }
  return RESS_OK;
}

int check_ws(const ress::Shape& s, void* ws, size_t ws_bytes, ress_ws_layout* L) {
  int e = check_ptr(ws, 256, "ws");
  if (e) return e;
  *L = ress::make_layout(s);
  if ((int64_t)ws_bytes < L->total)
    return fail(RESS_EWORKSPACE, "workspace has %zu bytes, needs %lld", ws_bytes, (long long)L->total);
  return RESS_OK;
}

int cuda_fail(cudaError_t e, const char* where) {
  return fail(RESS_ECUDA, "%s: %s", where, cudaGetErrorString(e));
}

// Streams and events the host-buffer forward owns: a second compute stream (the attention
// runs as chunks of query rows that alternate between it and the caller's stream, so that a
// chunk's CTAs take the SMs the previous chunk frees at its tail) and a copy stream that
// brings each chunk's output rows to the host while later chunks compute.  Created once per
// device on first use (never device memory); every call enqueues under one mutex because
// it re-records the same events.
constexpr int kOutChunks = 8;
constexpr int kMaxDevices = 64;
struct OverlapStreams {
  cudaStream_t aux = nullptr, copy = nullptr;
  cudaEvent_t ready = nullptr, copied = nullptr, done[kOutChunks] = {};
};
std::mutex g_overlap_mu;
OverlapStreams g_overlap[kMaxDevices];

cudaError_t overlap_streams(OverlapStreams** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  OverlapStreams& o = g_overlap[dev];
  if (!o.copied) {
    OverlapStreams n;
    if ((e = cudaStreamCreateWithFlags(&n.aux, cudaStreamNonBlocking)) != cudaSuccess ||
        (e = cudaStreamCreateWithFlags(&n.copy, cudaStreamNonBlocking)) != cudaSuccess ||
        (e = cudaEventCreateWithFlags(&n.ready, cudaEventDisableTiming)) != cudaSuccess)
      return e;
    for (int c = 0; c < kOutChunks; ++c)
      if ((e = cudaEventCreateWithFlags(&n.done[c], cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&n.copied, cudaEventDisableTiming)) != cudaSuccess) return e;
    o = n;
  }
  *out = &o;
  return cudaSuccess;
}

// col_idx entries of one head: every candidate query block keeps c_h candidates plus the
// always-kept key blocks, every other query block keeps all key blocks.
int64_t head_rows(const ress::Shape& s, int c) {
  const int nsk = s.nb - s.ncand;
  return (int64_t)s.nqc * (c + nsk) + (int64_t)(s.nq - s.nqc) * s.nb;
}

void head_bases(const ress::Shape& s, const int32_t* c, int64_t* base) {
  base[0] = 0;
  for (int h = 0; h < s.H; ++h) base[h + 1] = base[h] + head_rows(s, c[h]);
}

ress::SelectArgs select_args(const ress::Shape& s, const uint16_t* Q, const uint16_t* K,
                             const uint16_t* V, const float* F, const int32_t* c, void* ws,
                             const ress_ws_layout& L) {
  ress::SelectArgs a;
  a.s = s;
  a.Q = Q;
  a.K = K;
  a.V = V;
  a.F = F;
  a.ws = static_cast<char*>(ws);
  a.L = L;
  for (int h = 0; h < RESS_MAX_HEADS; ++h) a.c[h] = (c && h < s.H) ? c[h] : 0;
  a.v = ress::Variant{0, 0, 0ull, 0.0f};
  return a;
}

// NULL -> ReSS; otherwise the variant after a range check.
int check_variant(const ress_variant* v, ress::Variant* out) {
  *out = ress::Variant{0, 0, 0ull, 0.0f};
  if (!v) return RESS_OK;
  if (v->key < RESS_KEY_DRIFT || v->key > RESS_KEY_RANDOM)
    return fail(RESS_EINVAL, "variant key %d unknown", v->key);
  if (v->direction < RESS_MINIMIZE || v->direction > RESS_MAXIMIZE_FULL)
    return fail(RESS_EINVAL, "variant direction %d unknown", v->direction);
  if (!(v->cdf >= 0.0f && v->cdf <= 1.0f))
    return fail(RESS_EINVAL, "variant cdf %g outside [0, 1]", (double)v->cdf);
  if (v->cdf > 0.0f && v->direction != RESS_MINIMIZE)
    return fail(RESS_EINVAL, "a CDF threshold needs direction RESS_MINIMIZE");
  if (v->reserved != 0) return fail(RESS_EINVAL, "variant reserved field is %d, not 0", v->reserved);
  *out = ress::Variant{v->key, v->direction, (unsigned long long)v->seed, v->cdf};
  return RESS_OK;
}

}  // namespace

namespace ress {
void note_launch() { g_kernel_launches.fetch_add(1, std::memory_order_relaxed); }
cudaError_t launch_wait_selftest(uint32_t* status, uint64_t limit_ns, cudaStream_t st);  // k_select.cu
}  // namespace ress

extern "C" {

const char* ress_last_error(void) { return g_err; }

int32_t ress_abi_version(void) { return RESS_ABI_VERSION; }

uint64_t ress_kernel_launches(void) { return g_kernel_launches.load(std::memory_order_relaxed); }

int32_t ress_num_blocks(const ress_dims* d) {
  if (check_dims(d)) return -1;
  return ress::make_shape(*d).nb;
}

int32_t ress_num_candidates(const ress_dims* d) {
  if (check_dims(d)) return -1;
  return ress::make_shape(*d).ncand;
}
int32_t ress_num_query_blocks(const ress_dims* d) {
  if (check_dims(d)) return -1;
  return ress::make_shape(*d).nq;
}
int32_t ress_num_query_candidates(const ress_dims* d) {
  if (check_dims(d)) return -1;
  return ress::make_shape(*d).nqc;
}

size_t ress_workspace_bytes(const ress_dims* d) {
  if (check_dims(d)) return 0;
  return (size_t)ress::make_layout(ress::make_shape(*d)).total;
}

int ress_workspace_layout(const ress_dims* d, ress_ws_layout* out) {
  int e = check_dims(d);
  if (e) return e;
  if (!out) return fail(RESS_EINVAL, "out is NULL");
  *out = ress::make_layout(ress::make_shape(*d));
  return ok();
}

int64_t ress_csr_capacity(const ress_dims* d, const int32_t* c) {
  if (check_dims(d)) return -1;
  const ress::Shape s = ress::make_shape(*d);
  if (check_budgets(s, c)) return -1;
  int64_t base[RESS_MAX_HEADS + 1];
  head_bases(s, c, base);
  return base[s.H];
}

int64_t ress_csr_capacity_variant(const ress_dims* d, const int32_t* c, const ress_variant* v) {
  if (check_dims(d)) return -1;
  const ress::Shape s = ress::make_shape(*d);
  if (check_budgets(s, c)) return -1;
  ress::Variant var;
  if (check_variant(v, &var)) return -1;
  if (var.cdf > 0.0f) return (int64_t)s.H * s.nq * s.nb;
  int64_t base[RESS_MAX_HEADS + 1];
  head_bases(s, c, base);
  return base[s.H];
}

int ress_prepare_wo(const ress_dims* d, const uint16_t* W_o, float* F, void* stream) {
  int e = check_dims(d);
  if (e) return e;
  if ((e = check_ptr(W_o, 2, "W_o")) || (e = check_ptr(F, 16, "F"))) return e;
  const ress::Shape s = ress::make_shape(*d);
  cudaError_t ce = ress::launch_prepare_wo(s, W_o, F, static_cast<cudaStream_t>(stream));
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_prepare_wo");
  return ok();
}

int ress_score_variant(const ress_dims* d, const uint16_t* Q, const uint16_t* K,
                       const uint16_t* V, const float* F, const int32_t* c_h,
                       const ress_variant* variant, void* ws, size_t ws_bytes, void* stream) {
  int e = check_dims(d);
  if (e) return e;
  if ((e = check_ptr(Q, 16, "Q")) || (e = check_ptr(K, 16, "K")) || (e = check_ptr(V, 16, "V")) ||
      (e = check_ptr(F, 16, "F")))
    return e;
  const ress::Shape s = ress::make_shape(*d);
  if ((e = check_budgets(s, c_h))) return e;
  ress_ws_layout L;
  if ((e = check_ws(s, ws, ws_bytes, &L))) return e;
  ress::SelectArgs a = select_args(s, Q, K, V, F, c_h, ws, L);
  if ((e = check_variant(variant, &a.v))) return e;
  cudaError_t ce = ress::launch_score(a, static_cast<cudaStream_t>(stream));
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_score");
  return ok();
}

int ress_score(const ress_dims* d, const uint16_t* Q, const uint16_t* K, const uint16_t* V,
               const float* F, const int32_t* c_h, void* ws, size_t ws_bytes, void* stream) {
  return ress_score_variant(d, Q, K, V, F, c_h, nullptr, ws, ws_bytes, stream);
}

}  // extern "C"

// The restoration rounds and the CSR; with items set, the CSR kernel also writes the
// attention items' union lists into the workspace (a forward then skips k_pairs).
static int restore_impl(const ress_dims* d, const int32_t* c_h, int32_t rounds, float rho,
                        const ress_variant* variant, void* ws, size_t ws_bytes, int32_t* row_ptr,
                        int32_t* col_idx, int64_t col_capacity, float* J_best,
                        uint32_t* drop_mask, bool items, void* stream) {
  int e = check_dims(d);
  if (e) return e;
  const ress::Shape s = ress::make_shape(*d);
  if ((e = check_budgets(s, c_h))) return e;
  if (rounds < 0 || rounds > 32) return fail(RESS_EINVAL, "rounds %d outside 0..32", rounds);
  if (!(rho >= 0.0f && rho <= 1.0f)) return fail(RESS_EINVAL, "rho %g outside [0, 1]", (double)rho);
  ress_ws_layout L;
  if ((e = check_ws(s, ws, ws_bytes, &L))) return e;
  if ((e = check_ptr(row_ptr, 4, "row_ptr")) || (e = check_ptr(col_idx, 4, "col_idx"))) return e;
  if (J_best && (e = check_ptr(J_best, 4, "J_best"))) return e;
  if (drop_mask && (e = check_ptr(drop_mask, 4, "drop_mask"))) return e;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  ress::SelectArgs a = select_args(s, nullptr, nullptr, nullptr, nullptr, c_h, ws, L);
  if ((e = check_variant(variant, &a.v))) return e;
  if (a.v.cdf > 0.0f && rounds != 0)
    return fail(RESS_EINVAL, "a CDF threshold is defined without restoration rounds (rounds %d)", rounds);
  int64_t base[RESS_MAX_HEADS + 1];
  head_bases(s, c_h, base);
  // a CDF threshold may keep every key block of every row; the lists are written then at
  // the offsets of a device-side scan of the kept counts
  const int64_t need = a.v.cdf > 0.0f ? (int64_t)s.H * s.nq * s.nb : base[s.H];
  if (col_capacity < need)
    return fail(RESS_EWORKSPACE, "col_capacity %lld < %lld", (long long)col_capacity, (long long)need);
  if (need > INT32_MAX) return fail(RESS_EUNSUPPORTED, "CSR larger than 2^31 entries");
  for (int r = 0; r < rounds; ++r) {
    cudaError_t ce = ress::launch_round(a, r, rho, st);
    if (ce != cudaSuccess) return cuda_fail(ce, "ress_restore round");
  }
  char* w = static_cast<char*>(ws);
  int32_t* plist = items ? reinterpret_cast<int32_t*>(w + L.t) : nullptr;  // t is free by now
  int32_t* plen = items ? reinterpret_cast<int32_t*>(w + L.plen) : nullptr;
  // a forward pairs the query blocks of its attention items by the overlap of their kept lists
  int32_t* prow = nullptr;
  if (items && ress::pairing_active(s, a.v)) {
    prow = reinterpret_cast<int32_t*>(w + L.prow);
    cudaError_t ce = ress::launch_pairing(a, prow, st);
    if (ce != cudaSuccess) return cuda_fail(ce, "ress_restore pairing");
  }
  cudaError_t ce = ress::launch_csr(a, base, row_ptr, col_idx, col_capacity, J_best, drop_mask,
                                    plist, plen, (int64_t)s.H * s.nq * s.ld, prow, st);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_restore csr");
  return ok();
}

extern "C" {

int ress_restore_variant(const ress_dims* d, const int32_t* c_h, int32_t rounds, float rho,
                         const ress_variant* variant, void* ws, size_t ws_bytes, int32_t* row_ptr,
                         int32_t* col_idx, int64_t col_capacity, float* J_best,
                         uint32_t* drop_mask, void* stream) {
  return restore_impl(d, c_h, rounds, rho, variant, ws, ws_bytes, row_ptr, col_idx, col_capacity,
                      J_best, drop_mask, false, stream);
}

int ress_restore(const ress_dims* d, const int32_t* c_h, int32_t rounds, float rho, void* ws,
                 size_t ws_bytes, int32_t* row_ptr, int32_t* col_idx, int64_t col_capacity,
                 float* J_best, uint32_t* drop_mask, void* stream) {
  return ress_restore_variant(d, c_h, rounds, rho, nullptr, ws, ws_bytes, row_ptr, col_idx,
                              col_capacity, J_best, drop_mask, stream);
}

static ress::AttnArgs attn_args(const ress::Shape& s, const ress_ws_layout& L,
                                const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                                const int32_t* row_ptr, const int32_t* col_idx,
                                int64_t col_capacity, void* O, bool out_f32, void* ws) {
  char* w = static_cast<char*>(ws);
  ress::AttnArgs a;
  a.s = s;
  a.Q = Q;
  a.K = K;
  a.V = V;
  a.row_ptr = row_ptr;
  a.col_idx = col_idx;
  a.col_capacity = col_capacity;
  a.O = O;
  a.out_f32 = out_f32;
  a.status = reinterpret_cast<uint32_t*>(w + L.status);
  a.counter = reinterpret_cast<uint32_t*>(w + L.counter);
  a.plist = reinterpret_cast<int32_t*>(w + L.t);  // the gains buffer is free during attention
  a.plen = reinterpret_cast<int32_t*>(w + L.plen);
  a.scratch_cap = (int64_t)s.H * s.nq * s.ld;  // entries of the t array
  a.prow = nullptr;  // adjacent query blocks; a forward sets its pairing table
  a.npaired = 0;
  return a;
}

// The attention of a forward uses the item table its CSR step wrote (ReSS, no variant).
static void use_forward_pairing(ress::AttnArgs* a, const ress::Shape& s, const ress_ws_layout& L,
                                void* ws) {
  if (ress::pairing_active(s, ress::Variant{0, 0, 0ull, 0.0f})) {
    a->prow = reinterpret_cast<const int32_t*>(static_cast<char*>(ws) + L.prow);
    a->npaired = ress::paired_items(s);
  }
}

static int sparse_attn_impl(const ress_dims* d, const uint16_t* Q, const uint16_t* K,
                            const uint16_t* V, const int32_t* row_ptr, const int32_t* col_idx,
                            int64_t col_capacity, void* O, bool out_f32, void* ws, size_t ws_bytes,
                            void* stream) {
  int e = check_dims(d);
  if (e) return e;
  if ((e = check_ptr(Q, 16, "Q")) || (e = check_ptr(K, 16, "K")) || (e = check_ptr(V, 16, "V")) ||
      (e = check_ptr(O, 16, "O")) || (e = check_ptr(row_ptr, 4, "row_ptr")) ||
      (e = check_ptr(col_idx, 4, "col_idx")))
    return e;
  if (col_capacity < 0) return fail(RESS_EINVAL, "col_capacity %lld < 0", (long long)col_capacity);
  const ress::Shape s = ress::make_shape(*d);
  ress_ws_layout L;
  if ((e = check_ws(s, ws, ws_bytes, &L))) return e;
  const ress::AttnArgs a = attn_args(s, L, Q, K, V, row_ptr, col_idx, col_capacity, O, out_f32, ws);
  cudaError_t ce = ress::launch_sparse_attn(a, static_cast<cudaStream_t>(stream));
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_sparse_attn");
  return ok();
}

int ress_sparse_attn(const ress_dims* d, const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                     const int32_t* row_ptr, const int32_t* col_idx, int64_t col_capacity,
                     uint16_t* O, void* ws, size_t ws_bytes, void* stream) {
  return sparse_attn_impl(d, Q, K, V, row_ptr, col_idx, col_capacity, O, false, ws, ws_bytes, stream);
}

int ress_sparse_attn_f32(const ress_dims* d, const uint16_t* Q, const uint16_t* K,
                         const uint16_t* V, const int32_t* row_ptr, const int32_t* col_idx,
                         int64_t col_capacity, float* O, void* ws, size_t ws_bytes, void* stream) {
  return sparse_attn_impl(d, Q, K, V, row_ptr, col_idx, col_capacity, O, true, ws, ws_bytes, stream);
}

int ress_forward(const ress_dims* d, const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                 const float* F, const int32_t* c_h, int32_t rounds, float rho, void* ws,
                 size_t ws_bytes, int32_t* row_ptr, int32_t* col_idx, int64_t col_capacity,
                 uint16_t* O, float* J_best, void* stream) {
  // validate everything the three stages need before the first launch
  int e = check_dims(d);
  if (e) return e;
  if ((e = check_ptr(O, 16, "O"))) return e;
  const ress::Shape s = ress::make_shape(*d);
  if ((e = check_budgets(s, c_h))) return e;
  if (rounds < 0 || rounds > 32) return fail(RESS_EINVAL, "rounds %d outside 0..32", rounds);
  if (!(rho >= 0.0f && rho <= 1.0f)) return fail(RESS_EINVAL, "rho %g outside [0, 1]", (double)rho);
  if ((e = check_ptr(row_ptr, 4, "row_ptr")) || (e = check_ptr(col_idx, 4, "col_idx"))) return e;
  if (J_best && (e = check_ptr(J_best, 4, "J_best"))) return e;
  int64_t base[RESS_MAX_HEADS + 1];
  head_bases(s, c_h, base);
  if (col_capacity < base[s.H])
    return fail(RESS_EWORKSPACE, "col_capacity %lld < %lld", (long long)col_capacity, (long long)base[s.H]);
  ress_ws_layout L;
  if ((e = check_ws(s, ws, ws_bytes, &L))) return e;
  if ((e = ress_score(d, Q, K, V, F, c_h, ws, ws_bytes, stream))) return e;
  // the CSR kernel also writes the attention items' lists, so the attention starts directly
  if ((e = restore_impl(d, c_h, rounds, rho, nullptr, ws, ws_bytes, row_ptr, col_idx, col_capacity,
                        J_best, nullptr, true, stream)))
    return e;
  ress::AttnArgs a = attn_args(s, L, Q, K, V, row_ptr, col_idx, col_capacity, O, false, ws);
  use_forward_pairing(&a, s, L, ws);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t ce = cudaMemsetAsync(a.counter, 0, sizeof(uint32_t), st);
  if (ce == cudaSuccess) ce = ress::launch_attn_range(a, 0, ress::attn_num_pairs(s), 0, st);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_forward attention");
  return ok();
}

int ress_forward_host(const ress_dims* d, const uint16_t* Q_host, const uint16_t* K_host,
                      const uint16_t* V_host, uint16_t* O_host, uint16_t* Q_dev, uint16_t* K_dev,
                      uint16_t* V_dev, uint16_t* O_dev, const float* F, const int32_t* c_h,
                      int32_t rounds, float rho, void* ws, size_t ws_bytes, int32_t* row_ptr,
                      int32_t* col_idx, int64_t col_capacity, float* J_best, void* stream) {
  int e = check_dims(d);
  if (e) return e;
  if (!Q_host || !K_host || !V_host || !O_host) return fail(RESS_EINVAL, "null host buffer");
  if ((e = check_ptr(Q_dev, 16, "Q_dev")) || (e = check_ptr(K_dev, 16, "K_dev")) ||
      (e = check_ptr(V_dev, 16, "V_dev")) || (e = check_ptr(O_dev, 16, "O_dev")))
    return e;
  const size_t bytes = (size_t)d->n_tokens * (size_t)d->n_heads * 64 * sizeof(uint16_t);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // the forward's own checks run before any copy is enqueued: a dry validation first
  {
    const ress::Shape s = ress::make_shape(*d);
    if ((e = check_budgets(s, c_h))) return e;
    if (rounds < 0 || rounds > 32) return fail(RESS_EINVAL, "rounds %d outside 0..32", rounds);
    if (!(rho >= 0.0f && rho <= 1.0f)) return fail(RESS_EINVAL, "rho %g outside [0, 1]", (double)rho);
    if ((e = check_ptr(row_ptr, 4, "row_ptr")) || (e = check_ptr(col_idx, 4, "col_idx"))) return e;
    if (J_best && (e = check_ptr(J_best, 4, "J_best"))) return e;
    ress_ws_layout L;
    if ((e = check_ws(s, ws, ws_bytes, &L))) return e;
    int64_t base[RESS_MAX_HEADS + 1];
    head_bases(s, c_h, base);
    if (col_capacity < base[s.H])
      return fail(RESS_EWORKSPACE, "col_capacity %lld < %lld", (long long)col_capacity, (long long)base[s.H]);
  }
  const uint16_t* src[3] = {Q_host, K_host, V_host};
  uint16_t* dst[3] = {Q_dev, K_dev, V_dev};
  for (int k = 0; k < 3; ++k) {  // one copy per tensor
    cudaError_t ce = cudaMemcpyAsync(dst[k], src[k], bytes, cudaMemcpyHostToDevice, st);
    if (ce != cudaSuccess) return cuda_fail(ce, "ress_forward_host input copy");
  }
  if ((e = ress_score(d, Q_dev, K_dev, V_dev, F, c_h, ws, ws_bytes, stream))) return e;
  if ((e = restore_impl(d, c_h, rounds, rho, nullptr, ws, ws_bytes, row_ptr, col_idx, col_capacity,
                        J_best, nullptr, true, stream)))
    return e;
  // attention in chunks of 128-token query rows; each chunk's output rows go to the host on
  // the copy stream as soon as the chunk is done, while the next chunks compute
  const ress::Shape s = ress::make_shape(*d);
  ress_ws_layout L;
  if ((e = check_ws(s, ws, ws_bytes, &L))) return e;
  ress::AttnArgs a =
      attn_args(s, L, Q_dev, K_dev, V_dev, row_ptr, col_idx, col_capacity, O_dev, false, ws);
  use_forward_pairing(&a, s, L, ws);
  std::lock_guard<std::mutex> lock(g_overlap_mu);
  OverlapStreams* o = nullptr;
  cudaError_t ce = overlap_streams(&o);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_forward_host streams");
  if ((ce = cudaMemsetAsync(a.counter, 0, kOutChunks * sizeof(uint32_t), st)) != cudaSuccess ||
      (ce = cudaEventRecord(o->ready, st)) != cudaSuccess ||
      (ce = cudaStreamWaitEvent(o->aux, o->ready, 0)) != cudaSuccess)
    return cuda_fail(ce, "ress_forward_host attention");
  const int np = ress::attn_num_pairs(s);
  const int chunks = np < kOutChunks ? np : kOutChunks;
  const size_t row_bytes = bytes / (size_t)d->n_tokens;  // one token: H * 64 bf16
  // chunk boundaries among the paired items fall on whole pairing windows, so that every
  // chunk's items hold exactly the query rows [128 p0, 128 p1)
  auto bound = [&](int c) {
    int b = (int)((int64_t)np * c / chunks);
    if (b < a.npaired) b = b / (ress::kPairWindow / 2) * (ress::kPairWindow / 2);
    return b;
  };
  for (int c = 0; c < chunks && ce == cudaSuccess; ++c) {
    const int p0 = bound(c), p1 = c + 1 == chunks ? np : bound(c + 1);
    if (p1 <= p0) continue;
    cudaStream_t cs = (c & 1) ? o->aux : st;
    const int64_t t0 = 128 * (int64_t)p0;
    const int64_t t1 = 128 * (int64_t)p1 < d->n_tokens ? 128 * (int64_t)p1 : d->n_tokens;
    if ((ce = ress::launch_attn_range(a, p0, p1, c, cs)) == cudaSuccess &&
        (ce = cudaEventRecord(o->done[c], cs)) == cudaSuccess &&
        (ce = cudaStreamWaitEvent(o->copy, o->done[c], 0)) == cudaSuccess)
      ce = cudaMemcpyAsync(reinterpret_cast<char*>(O_host) + t0 * row_bytes,
                           reinterpret_cast<const char*>(O_dev) + t0 * row_bytes,
                           (size_t)(t1 - t0) * row_bytes, cudaMemcpyDeviceToHost, o->copy);
  }
  // the caller's stream resumes after every chunk and copy (also after a failed enqueue)
  cudaError_t je = cudaEventRecord(o->copied, o->copy);
  if (je == cudaSuccess) je = cudaStreamWaitEvent(st, o->copied, 0);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_forward_host attention chunk");
  if (je != cudaSuccess) return cuda_fail(je, "ress_forward_host join");
  return ok();
}

int ress_wait_selftest(void* ws, size_t ws_bytes, uint32_t limit_us, void* stream) {
  int e = check_ptr(ws, 256, "ws");
  if (e) return e;
  if (ws_bytes < 64) return fail(RESS_EWORKSPACE, "workspace has %zu bytes, needs 64", ws_bytes);
  if (limit_us < 1 || limit_us > 100000)
    return fail(RESS_EINVAL, "limit_us %u outside 1..100000", limit_us);
  cudaError_t ce = ress::launch_wait_selftest(static_cast<uint32_t*>(ws), 1000ull * limit_us,
                                              static_cast<cudaStream_t>(stream));
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_wait_selftest");
  return ok();
}

int ress_status(void* ws, void* stream) {
  int e = check_ptr(ws, 256, "ws");
  if (e) return e;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t ce = cudaStreamSynchronize(st);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_status sync");
  uint32_t word = 0;
  ce = cudaMemcpy(&word, ws, sizeof(word), cudaMemcpyDeviceToHost);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_status read");
  ce = cudaMemset(ws, 0, sizeof(word));
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_status clear");
  if (word == 0) return ok();
  if (word == ress::kStatusTimeout) return fail(RESS_ETIMEOUT, "a bounded device wait gave up");
  return fail(RESS_EDEVICE, "device-side argument check failed (code %u)", word);
}

static int oproj_checks(const ress_dims* d, const void* W_o, void* ws, size_t ws_bytes,
                        ress::Shape* s, ress_ws_layout* L) {
  int e = check_dims(d);
  if (e) return e;
  if ((e = check_ptr(W_o, 16, "W_o"))) return e;
  if (d->d_model % 64 != 0)
    return fail(RESS_EUNSUPPORTED, "d_model %d must be a multiple of 64", d->d_model);
  *s = ress::make_shape(*d);
  return check_ws(*s, ws, ws_bytes, L);
}

int ress_out_proj(const ress_dims* d, const uint16_t* O, const uint16_t* W_o, const uint16_t* x,
                  uint16_t* y, void* ws, size_t ws_bytes, void* stream) {
  ress::Shape s{};
  ress_ws_layout L{};
  int e = oproj_checks(d, W_o, ws, ws_bytes, &s, &L);
  if (e) return e;
  if ((e = check_ptr(O, 16, "O")) || (e = check_ptr(y, 16, "y"))) return e;
  if (x && (e = check_ptr(x, 16, "x"))) return e;
  ress::OProjArgs a;
  a.N = s.N;
  a.H = s.H;
  a.Dm = d->d_model;
  a.O = O;
  a.O2 = nullptr;
  a.W_o = W_o;
  a.x = x;
  a.y = y;
  a.drift = nullptr;
  a.status = reinterpret_cast<uint32_t*>(static_cast<char*>(ws) + L.status);
  cudaError_t ce = ress::launch_out_proj(a, static_cast<cudaStream_t>(stream));
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_out_proj");
  return ok();
}

int ress_token_drift(const ress_dims* d, const uint16_t* O_a, const uint16_t* O_b,
                     const uint16_t* W_o, float* drift, void* ws, size_t ws_bytes, void* stream) {
  ress::Shape s{};
  ress_ws_layout L{};
  int e = oproj_checks(d, W_o, ws, ws_bytes, &s, &L);
  if (e) return e;
  if ((e = check_ptr(O_a, 16, "O_a")) || (e = check_ptr(O_b, 16, "O_b")) ||
      (e = check_ptr(drift, 4, "drift")))
    return e;
  ress::OProjArgs a;
  a.N = s.N;
  a.H = s.H;
  a.Dm = d->d_model;
  a.O = O_a;
  a.O2 = O_b;
  a.W_o = W_o;
  a.x = nullptr;
  a.y = nullptr;
  a.drift = drift;
  a.status = reinterpret_cast<uint32_t*>(static_cast<char*>(ws) + L.status);
  cudaError_t ce = ress::launch_token_drift(a, static_cast<cudaStream_t>(stream));
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_token_drift");
  return ok();
}

}  // extern "C"

// ---------------------------------------------------------------------------------------
// Allocation-free attention entry point.
//
// Some callers cannot allocate device memory when they call into this library: a host
// framework that owns every byte of device memory through its own pool and forbids
// allocations inside plugins, a real-time runtime that reserves all memory at start-up
// because a later cudaMalloc can stall the device and may fail under a tight budget, or a
// caller that cannot spare the full ress workspace just for the attention step.  For them
// this entry point keeps its scratch (status word, tile counter, pair lengths and pair
// lists) in a file-scope __device__ array of RESS_NOALLOC_SCRATCH_BYTES that every GPU
// loading the library holds until the process exits.  The caller still passes Q, K, V, the
// CSR and O.
// ---------------------------------------------------------------------------------------
#include <mutex>

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[RESS_NOALLOC_SCRATCH_BYTES];

constexpr int kNoallocMaxDevices = 64;
constexpr int64_t kNoallocStatus = 0;    // uint32 status word
constexpr int64_t kNoallocCounter = 64;  // uint32 tile counter (zeroed by every launch)
constexpr int64_t kNoallocPlen = 256;    // int32 pair lengths, then the pair lists

std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kNoallocMaxDevices] = {};

// Device address of the scratch array on the current device.  In host code the array's
// name is only a host-side stand-in, so the address is looked up once per device (with
// that device current) and cached.
int noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t ce = cudaGetDevice(&dev);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_sparse_attn_noalloc: cudaGetDevice");
  if (dev < 0 || dev >= kNoallocMaxDevices)
    return fail(RESS_EUNSUPPORTED, "device ordinal %d beyond %d", dev, kNoallocMaxDevices);
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    ce = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (ce != cudaSuccess || !p) return cuda_fail(ce, "ress_sparse_attn_noalloc: cudaGetSymbolAddress");
    g_noalloc_ptr[dev] = p;
  }
  *out = g_noalloc_ptr[dev];
  return RESS_OK;
}

}  // namespace

extern "C" int ress_sparse_attn_noalloc(const ress_dims* d, const uint16_t* Q, const uint16_t* K,
                                        const uint16_t* V, const int32_t* row_ptr,
                                        const int32_t* col_idx, int64_t col_capacity, uint16_t* O,
                                        int32_t wait, void* stream) {
  int e = check_dims(d);
  if (e) return e;
  if ((e = check_ptr(Q, 16, "Q")) || (e = check_ptr(K, 16, "K")) || (e = check_ptr(V, 16, "V")) ||
      (e = check_ptr(O, 16, "O")) || (e = check_ptr(row_ptr, 4, "row_ptr")) ||
      (e = check_ptr(col_idx, 4, "col_idx")))
    return e;
  if (col_capacity < 0) return fail(RESS_EINVAL, "col_capacity %lld < 0", (long long)col_capacity);
  const ress::Shape s = ress::make_shape(*d);
  const int64_t plen_bytes = ress::align256((int64_t)s.H * ((s.nb + 1) / 2) * 4);
  const int64_t list_entries = ((int64_t)RESS_NOALLOC_SCRATCH_BYTES - kNoallocPlen - plen_bytes) / 4;
  if (col_capacity > list_entries)
    return fail(RESS_EWORKSPACE,
                "col_capacity %lld exceeds the %lld CSR entries that the built-in %u-byte scratch "
                "holds for %d heads x %d blocks; use ress_sparse_attn with a workspace",
                (long long)col_capacity, (long long)list_entries, (unsigned)RESS_NOALLOC_SCRATCH_BYTES,
                s.H, s.nb);
  void* base = nullptr;
  if ((e = noalloc_scratch(&base))) return e;
  char* w = static_cast<char*>(base);
  ress::AttnArgs a;
  a.s = s;
  a.Q = Q;
  a.K = K;
  a.V = V;
  a.row_ptr = row_ptr;
  a.col_idx = col_idx;
  a.col_capacity = col_capacity;
  a.O = O;
  a.out_f32 = false;
  a.status = reinterpret_cast<uint32_t*>(w + kNoallocStatus);
  a.counter = reinterpret_cast<uint32_t*>(w + kNoallocCounter);
  a.plen = reinterpret_cast<int32_t*>(w + kNoallocPlen);
  a.plist = reinterpret_cast<int32_t*>(w + kNoallocPlen + plen_bytes);
  a.scratch_cap = list_entries;
  a.prow = nullptr;  // items of adjacent query blocks
  a.npaired = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t ce = ress::launch_sparse_attn(a, st);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_sparse_attn_noalloc");
  if (!wait) return ok();
  ce = cudaStreamSynchronize(st);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_sparse_attn_noalloc sync");
  uint32_t word = 0;
  ce = cudaMemcpy(&word, a.status, sizeof(word), cudaMemcpyDeviceToHost);
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_sparse_attn_noalloc status read");
  if (word == 0) return ok();
  ce = cudaMemset(a.status, 0, sizeof(word));
  if (ce != cudaSuccess) return cuda_fail(ce, "ress_sparse_attn_noalloc status clear");
  if (word == ress::kStatusTimeout) return fail(RESS_ETIMEOUT, "a bounded device wait gave up");
  return fail(RESS_EDEVICE, "device-side argument check failed (code %u)", word);
}
