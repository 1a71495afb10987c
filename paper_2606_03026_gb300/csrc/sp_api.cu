// sp_api.cu -- the C ABI of libspikeproj.so: argument validation, plans and
// groups (workspace ownership), per-call dispatch between the gather, union
// and tensor-core kernels, and status reporting.  See include/spike_proj.h.
#include <atomic>
#include <cstdlib>
#include <algorithm>
#include <cstring>
#include <mutex>
#include <new>

#include "sp_gemm.h"
#include "sp_internal.h"

using namespace sp;

// Scratch of spike_proj_decode_noalloc, one copy per device in static device
// memory: the split-K workspace of one spike row at the largest N and one
// ticket per 512-channel output tile.  Zero when the module loads; every
// gather launch that completes leaves it zero (the kernel has no error path:
// no waits, no aborts), so no call has to clear it.
constexpr int kNoallocMaxN = SPIKE_PROJ_NOALLOC_MAX_N;
constexpr int kNoallocTickets = kNoallocMaxN / kGatherNT;
constexpr int kNoallocWords = kNoallocMaxN + kNoallocTickets;
static_assert(kNoallocMaxN % kGatherNT == 0, "whole output tiles");
static __device__ __align__(256) int32_t g_noalloc_scratch[kNoallocWords];

struct sp_plan_s {
  int device = 0;
  const int8_t* W = nullptr;
  int64_t ldw = 0;
  const float* scale = nullptr;
  int32_t N = 0, K = 0, max_batch = 0;
  uint32_t flags = 0;
  int32_t* ws = nullptr;          // [max_batch][N] INT32, zero between calls
  uint32_t* tickets = nullptr;    // zero between calls
  size_t n_tickets = 0;
  int* err = nullptr;             // device error word
  int32_t* d_counts = nullptr;    // density probe result [2]
  int32_t* h_counts = nullptr;    // page-locked copy
  // tensor-core path
  uint8_t* Wq = nullptr;          // [N][2 Kp] e4m3 weight planes (16 h, l)
  uint8_t* Xs = nullptr;          // [xs_rows][Kp] 0/1 spike staging
  float* part = nullptr;          // split-K partials, part_units x 128 x 256 fp32
  int Kp = 0, xs_rows = 0, part_units = 0;
  GemmMaps maps;
  CUtensorMap rows_map;           // caller's 0/1 rows of the last in-place call
  const void* rows_ptr = nullptr;
  int64_t rows_ld = 0;
  int32_t rows_T = 0;
  sp_kernel last_kernel = SP_AUTO;
  int32_t last_active = -1;
  int32_t fault = 0;              // test fault armed for the next launch (sp_fault)
};

struct sp_head_s {
  int device = 0;
  const int8_t* W = nullptr;
  int64_t ldw = 0;
  const float* scale = nullptr;
  int32_t V = 0, K = 0;
  uint8_t* ws = nullptr;          // head_workspace_bytes()
};

struct sp_group_s {
  int32_t count = 0;
  int32_t maxN = 0, maxK = 0;
  GatherParamsG params;           // problem table, per-call fields filled in at each call
  int32_t* ws = nullptr;
  uint32_t* tickets = nullptr;
  int* err = nullptr;
  size_t ws_elems = 0, n_tickets = 0;
  // staging for the host-buffer entry point
  void* d_spikes = nullptr;       // [count][row bytes]
  int32_t* d_acc = nullptr;       // [count][maxN]
  float* d_y = nullptr;           // [count][maxN]
  size_t spike_row_bytes = 0;
  // grouped prefill (every plan made with SP_PLAN_GEMM): the launch's member
  // table, and per member the caller's 0/1 rows of the last in-place call
  sp_plan_s* plans[kMaxProblems] = {};
  GemmGroupArgs* gemm = nullptr;
  float* gpart = nullptr;         // tail-split partials (groups of SP_PLAN_GEMM plans)
  uint32_t* gflags = nullptr;     // their flags, zero between launches
  int32_t fault = 0;              // test fault armed for the next launch (sp_fault)
  const void* rows_ptr[kMaxProblems] = {};
  int64_t rows_ld[kMaxProblems] = {};
  int32_t rows_T[kMaxProblems] = {};
  CUtensorMap rows_map[kMaxProblems];
};

namespace {

thread_local int g_last_cuda_error = 0;

inline sp_status cuda_fail(cudaError_t e) {
  g_last_cuda_error = (int)e;
  return SP_ECUDA;
}
#define SP_CUDA(call)                              \
  do {                                             \
    cudaError_t e_ = (call);                       \
    if (e_ != cudaSuccess) return cuda_fail(e_);   \
  } while (0)

inline bool aligned(const void* p, uintptr_t a) {
  return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0;
}
inline cudaStream_t as_stream(sp_stream_t s) { return reinterpret_cast<cudaStream_t>(s); }
inline int64_t words_for(int K) { return ((int64_t)K + 31) / 32; }
inline int64_t row_elems(sp_fmt fmt, int K) { return fmt == SP_SPIKES_BITS32 ? words_for(K) : K; }
inline bool fmt_ok(int fmt) {
  return fmt == SP_SPIKES_BITS32 || fmt == SP_SPIKES_U8 || fmt == SP_SPIKES_BOOL8;
}

sp_status check_device(int* dev_out) {
  int dev = 0, major = 0, minor = 0;
  SP_CUDA(cudaGetDevice(&dev));
  SP_CUDA(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev));
  SP_CUDA(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev));
  if (major != 10 || minor != 3) return SP_EDEVICE;
  *dev_out = dev;
  return SP_OK;
}

template <typename T>
sp_status dev_alloc_zero(T** p, size_t count, cudaStream_t s) {
  if (count == 0) count = 1;
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T));
  if (e != cudaSuccess) {
    *p = nullptr;
    g_last_cuda_error = (int)e;
    (void)cudaGetLastError();
    return e == cudaErrorMemoryAllocation ? SP_ENOMEM : SP_ECUDA;
  }
  SP_CUDA(cudaMemsetAsync(*p, 0, count * sizeof(T), s));
  return SP_OK;
}

void plan_free(sp_plan_s* p) {
  if (!p) return;
  cudaFree(p->ws);
  cudaFree(p->tickets);
  cudaFree(p->err);
  cudaFree(p->d_counts);
  if (p->h_counts) cudaFreeHost(p->h_counts);
  cudaFree(p->Wq);
  cudaFree(p->Xs);
  cudaFree(p->part);
  delete p;
}

void group_free(sp_group_s* g) {
  if (!g) return;
  delete g->gemm;
  cudaFree(g->gpart);
  cudaFree(g->gflags);
  cudaFree(g->ws);
  cudaFree(g->tickets);
  cudaFree(g->err);
  cudaFree(g->d_spikes);
  cudaFree(g->d_acc);
  cudaFree(g->d_y);
  delete g;
}

// Device address of page-locked host memory that the current device can
// reach (cudaHostAlloc, cudaHostRegister, torch pin_memory), else nullptr.
void* device_view(const void* h) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, h) != cudaSuccess) {
    (void)cudaGetLastError();
    return nullptr;
  }
  return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}

// Spike / output argument checks shared by the per-plan calls.
sp_status check_io(const void* spikes, int fmt, const int32_t* acc, const float* y) {
  if (!spikes || !fmt_ok(fmt)) return SP_EINVAL;
  if (!acc && !y) return SP_EINVAL;
  if (fmt == SP_SPIKES_BITS32 && !aligned(spikes, 4)) return SP_EALIGN;
  if ((acc && !aligned(acc, 4)) || (y && !aligned(y, 4))) return SP_EALIGN;
  return SP_OK;
}

GatherParams1 single_params(const sp_plan_s* p, const void* spikes, int fmt, int B, int64_t ld,
                            int32_t* acc, float* y) {
  GatherParams1 g;
  std::memset(&g, 0, sizeof(g));
  g.prob[0].W = p->W;
  g.prob[0].scale = p->scale;
  g.prob[0].ldw = (int32_t)p->ldw;
  g.prob[0].N = p->N;
  g.prob[0].K = p->K;
  g.nprob = 1;
  g.B = B;
  g.units_total = B * gather_units(p->N, p->K);
  g.max_units = gather_units(p->N, p->K);
  g.fmt = fmt;
  g.spikes = spikes;
  g.ld_spikes = ld;
  g.acc = acc;
  g.y = y;
  g.ld_out = p->N;
  g.ws = p->ws;
  g.tickets = p->tickets;
  g.err = p->err;
  return g;
}

// Several rows of one plan as a group of that many one-row problems sharing
// W: the group launch then runs them in the cluster form (each row's tiles x
// chunks in clusters, partials exchanged in shared memory) when every
// cluster can be resident at once, and in the ticket form otherwise.  The
// workspace and ticket offsets (row t: ws + t N, tickets + t ntiles) are the
// batched ticket form's, so the plan's workspace serves both.
GatherParamsG rows_as_group(const sp_plan_s* p, const void* spikes, int fmt, int B, int64_t ld,
                            int32_t* acc, float* y) {
  GatherParamsG g;
  std::memset(&g, 0, sizeof(g));
  const int units = gather_units(p->N, p->K);
  for (int t = 0; t < B; ++t) {
    GatherProblem& P = g.prob[t];
    P.W = p->W;
    P.scale = p->scale;
    P.ldw = (int32_t)p->ldw;
    P.N = p->N;
    P.K = p->K;
    P.unit_begin = t * units;
    P.ws_begin = t * p->N;
    P.ticket_begin = t * gather_ntiles(p->N);
  }
  g.nprob = B;
  g.B = 1;
  g.units_total = B * units;
  g.max_units = units;
  g.fmt = fmt;
  g.spikes = spikes;
  g.ld_spikes = ld;
  g.acc = acc;
  g.y = y;
  g.ld_out = p->N;
  g.ws = p->ws;
  g.tickets = p->tickets;
  g.err = p->err;
  return g;
}

sp_status run_gather(sp_plan_s* p, const void* spikes, int fmt, int B, int64_t ld, int32_t* acc,
                     float* y, cudaStream_t s) {
  if (B > 1 && B <= kMaxProblems && (int64_t)B * p->N <= INT32_MAX) {
    GatherParamsG g = rows_as_group(p, spikes, fmt, B, ld, acc, y);
    g.fault = p->fault;
    p->fault = 0;
    SP_CUDA(launch_gather(g, s));
    return SP_OK;
  }
  GatherParams1 g = single_params(p, spikes, fmt, B, ld, acc, y);
  g.fault = p->fault;
  p->fault = 0;
  SP_CUDA(launch_gather(g, s));
  return SP_OK;
}

sp_status run_union(sp_plan_s* p, const void* spikes, int fmt, int B, int64_t ld, int32_t* acc,
                    float* y, cudaStream_t s) {
  const int64_t elem = fmt == SP_SPIKES_BITS32 ? 4 : 1;
  for (int b0 = 0; b0 < B; b0 += kUnionMaxRows) {
    const int nb = B - b0 < kUnionMaxRows ? B - b0 : kUnionMaxRows;
    UnionParams u;
    u.W = p->W;
    u.scale = p->scale;
    u.ldw = (int32_t)p->ldw;
    u.N = p->N;
    u.K = p->K;
    u.B = nb;
    u.fmt = fmt;
    u.spikes = static_cast<const uint8_t*>(spikes) + (int64_t)b0 * ld * elem;
    u.ld_spikes = ld;
    u.acc = acc ? acc + (int64_t)b0 * p->N : nullptr;
    u.y = y ? y + (int64_t)b0 * p->N : nullptr;
    u.ws = p->ws;
    u.tickets = p->tickets;
    u.err = p->err;
    u.fault = p->fault;
    p->fault = 0;
    SP_CUDA(launch_union(u, s));
  }
  return SP_OK;
}

sp_status run_gemm(sp_plan_s* p, const void* spikes, int fmt, int T, int64_t ld, int32_t* acc,
                   float* y, cudaStream_t s) {
  if (!(p->flags & SP_PLAN_GEMM)) return SP_EUNSUPPORTED;
  // a few rows: the transposed small-T form reads the spike rows in place
  if (const int S = gemm_small_splits(T, p->N, p->Kp)) {
    GemmSmallArgs g;
    g.spikes = spikes;
    g.fmt = fmt;
    g.ld = ld;
    g.scale = p->scale;
    g.acc = acc;
    g.y = y;
    g.T = T;
    g.TN = ceil_div(T, 16) * 16;
    g.N = p->N;
    g.K = p->K;
    g.S = S;
    g.nkb = p->Kp / 64;
    g.err = p->err;
    g.fault = p->fault;
    p->fault = 0;
    SP_CUDA(launch_gemm_small(p->maps.p64, g, s));
    return SP_OK;
  }
  // 0/1 byte rows that TMA can address are the MMA's spike operand as they
  // stand; any other input is first written as 0/1 bytes into the staging copy
  const bool in_place = fmt == SP_SPIKES_BOOL8 && aligned(spikes, 16) && ld % 16 == 0;
  const int S = gemm_splits(T, p->N, p->Kp, p->part_units);
  if (in_place) {
    if (spikes != p->rows_ptr || ld != p->rows_ld || T != p->rows_T) {
      SP_CUDA(gemm_make_rows_map(spikes, ld, T, p->K, &p->rows_map));
      p->rows_ptr = spikes;
      p->rows_ld = ld;
      p->rows_T = T;
    }
  } else {
    SP_CUDA(launch_spikes_to_01(spikes, fmt, ld, T, p->K, p->Kp, p->Xs, s));
  }
  GemmParams g;
  g.scale = p->scale;
  g.acc = acc;
  g.y = y;
  g.T = T;
  g.N = p->N;
  g.K = p->K;
  g.err = p->err;
  g.part = p->part;
  g.part_units = p->part_units;
  g.fault = p->fault;
  p->fault = 0;
  SP_CUDA(launch_gemm(in_place ? p->rows_map : p->maps.a, p->maps.b, S, T, p->N, p->Kp, g, s));
  return SP_OK;
}

// Measured-density dispatch between the per-token gather and the
// tensor-core GEMM, by a cost model fitted on GB300 (token rates
// U(0.05, 0.2), weights L2-resident, graph-timed, N x K in {1536 x 6144,
// 1536 x 1536, 4096 x 1536, 1536 x 16384}, B = 1 .. 256):
//   gather        ~ 3.9 us + 0.08 us per row after the first
//                   + active bytes (sum_t |A_t| * N) / 6.7 TB/s
//   GEMM, T <= 64 ~ 3.4 us + 0.33 us per K block of a CTA's K range
//                   (ceil(Kp / 64 / S), S = the cluster size) + 0.045 us per row
//   GEMM, T > 64  ~ max(11.3 us + 2 B N K ops / 1.4 PFLOP/s, 8.5 us + 0.55 us per 1024 of K)
// (the GEMM only for SP_PLAN_GEMM plans).  Measured at 1536 x 6144: gather
// 4.2 / 6.7 / 9.0 / 11.6 / 16.5 us at B = 1 / 8 / 16 / 32 / 64 in the ticket
// form, and 6.0 / 7.6 / 9.3 us at B = 8 / 16 / 32 with the rows run as a
// group (the fixed term fitted to the latter: 4.2 us before), small-T GEMM
// 7.2 / 7.2 / 7.3 / 8.0 / 9.2 us, the 128-row GEMM 12.1 us at B = 65 .. 128
// (17.5 us at K = 16384); at 1536 x 1536 the gather (rows as a group) wins
// up to B = 6 (3.6 against 4.5 us at B = 4) and the small-T GEMM from B = 8.  The union fetch is never chosen automatically: it
// was slower than the per-token gather at every batch size measured (its
// adds are ALU-bound, and the 126 MB L2 serves the per-token re-reads of a
// 9.4 MB weight matrix).
sp_kernel choose(const sp_plan_s* p, int B, int32_t total) {
  if (!(p->flags & SP_PLAN_GEMM)) return SP_GATHER;
  const double gather_us = 3.9 + 0.08 * (B - 1) + (double)total * p->N / 6.7e6;
  double gemm_us;
  const int nkb = p->Kp / 64;
  if (const int S = gemm_small_splits(B, p->N, p->Kp))
    gemm_us = 3.4 + 0.33 * ceil_div(nkb, S) + 0.045 * B;
  else
    gemm_us = std::max(11.3 + 2.0 * B * (double)p->N * p->K / 1.4e9, 8.5 + 0.55 * p->K / 1024.0);
  return gemm_us < gather_us ? SP_GEMM : SP_GATHER;
}

sp_status run_multi(sp_plan_s* p, const void* spikes, int fmt, int B, int64_t ld, int32_t* acc,
                    float* y, sp_kernel strategy, cudaStream_t s) {
  if (strategy == SP_AUTO) {
    SP_CUDA(launch_density(spikes, fmt, ld, B, p->K, p->d_counts, s));
    SP_CUDA(cudaMemcpyAsync(p->h_counts, p->d_counts, 2 * sizeof(int32_t), cudaMemcpyDeviceToHost, s));
    SP_CUDA(cudaStreamSynchronize(s));
    strategy = choose(p, B, p->h_counts[0]);
    p->last_kernel = strategy;
    p->last_active = p->h_counts[0];
  }
  switch (strategy) {
    case SP_GATHER: return run_gather(p, spikes, fmt, B, ld, acc, y, s);
    case SP_UNION: return run_union(p, spikes, fmt, B, ld, acc, y, s);
    case SP_GEMM: return run_gemm(p, spikes, fmt, B, ld, acc, y, s);
    default: return SP_EINVAL;
  }
}

// Per-device address of g_noalloc_scratch, set once by the first call on the
// device (with that device current).  Later calls read it without a lock.
// The address belongs to the device's current context: after
// cudaDeviceReset the entry point must not be called again in this process.
constexpr int kNoallocDevices = 64;
std::mutex g_noalloc_mu;
std::atomic<int32_t*> g_noalloc_ptr[kNoallocDevices];

sp_status noalloc_scratch(cudaStream_t s, int32_t** out) {
  int dev = 0;
  SP_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kNoallocDevices) return SP_EDEVICE;
  int32_t* ptr = g_noalloc_ptr[dev].load(std::memory_order_acquire);
  if (!ptr) {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    ptr = g_noalloc_ptr[dev].load(std::memory_order_relaxed);
    if (!ptr) {
      int checked = 0;
      const sp_status st = check_device(&checked);
      if (st != SP_OK) return st;
      void* sym = nullptr;
      SP_CUDA(cudaGetSymbolAddress(&sym, g_noalloc_scratch));
      // defensive: the array is already zero when the module loads
      SP_CUDA(cudaMemsetAsync(sym, 0, sizeof(g_noalloc_scratch), s));
      SP_CUDA(cudaStreamSynchronize(s));
      ptr = static_cast<int32_t*>(sym);
      g_noalloc_ptr[dev].store(ptr, std::memory_order_release);
    }
  }
  *out = ptr;
  return SP_OK;
}

}  // namespace

// ============================================================================
extern "C" {

sp_status spike_proj_plan(sp_plan_t* plan, const int8_t* W, int64_t ldw, const float* scale,
                          int32_t N, int32_t K, int32_t max_batch, uint32_t flags,
                          sp_stream_t stream) {
  if (!plan || !W || !scale) return SP_EINVAL;
  if (N < 16 || max_batch < 1 || max_batch > (1 << 20)) return SP_EINVAL;
  if ((flags & ~SP_PLAN_GEMM) != 0) return SP_EINVAL;
  if (K < 1 || K > SPIKE_PROJ_MAX_K) return SP_ERANGE;
  if (N % 16 != 0 || ldw < N || ldw % 16 != 0 || ldw > INT32_MAX) return SP_EALIGN;
  if (!aligned(W, 16) || !aligned(scale, 4)) return SP_EALIGN;
  int dev = 0;
  sp_status st = check_device(&dev);
  if (st != SP_OK) return st;
  if ((int64_t)max_batch * N > ((int64_t)1 << 31)) return SP_ERANGE;

  cudaStream_t s = as_stream(stream);
  sp_plan_s* p = new (std::nothrow) sp_plan_s();
  if (!p) return SP_ENOMEM;
  p->device = dev;
  p->W = W;
  p->ldw = ldw;
  p->scale = scale;
  p->N = N;
  p->K = K;
  p->max_batch = max_batch;
  p->flags = flags;

  size_t tickets = (size_t)max_batch * gather_ntiles(N);
  const size_t union_t = (size_t)ceil_div(N, kUnionNT);
  if (union_t > tickets) tickets = union_t;
  p->n_tickets = tickets;
  if ((st = dev_alloc_zero(&p->ws, (size_t)max_batch * N, s)) != SP_OK ||
      (st = dev_alloc_zero(&p->tickets, tickets, s)) != SP_OK ||
      (st = dev_alloc_zero(&p->err, 1, s)) != SP_OK ||
      (st = dev_alloc_zero(&p->d_counts, 2, s)) != SP_OK) {
    plan_free(p);
    return st;
  }
  cudaError_t e = cudaMallocHost(reinterpret_cast<void**>(&p->h_counts), 2 * sizeof(int32_t));
  if (e != cudaSuccess) {
    plan_free(p);
    return cuda_fail(e);
  }
  if (flags & SP_PLAN_GEMM) {
    p->Kp = gemm_k_pad(K);
    p->xs_rows = ceil_div(max_batch, 128) * 128;
    // a split-K launch has at most one unit per SM
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) {
      plan_free(p);
      return cuda_fail(e);
    }
    p->part_units = sms;
    if ((st = dev_alloc_zero(&p->Wq, (size_t)2 * N * p->Kp, s)) != SP_OK ||
        (st = dev_alloc_zero(&p->Xs, (size_t)p->xs_rows * p->Kp, s)) != SP_OK ||
        (st = dev_alloc_zero(&p->part, (size_t)p->part_units * kGemmPartialElems, s)) != SP_OK) {
      plan_free(p);
      return st;
    }
    e = launch_w_to_e4m3(W, ldw, N, K, p->Wq, s);
    if (e == cudaSuccess) e = gemm_make_maps(p->Xs, p->xs_rows, p->Wq, N, p->Kp, &p->maps);
    if (e != cudaSuccess) {
      plan_free(p);
      return cuda_fail(e);
    }
  }
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    plan_free(p);
    return cuda_fail(e);
  }
  *plan = p;
  return SP_OK;
}

sp_status spike_proj_plan_destroy(sp_plan_t plan) {
  if (!plan) return SP_OK;
  cudaError_t e = cudaDeviceSynchronize();
  plan_free(plan);
  return e == cudaSuccess ? SP_OK : cuda_fail(e);
}

sp_status spike_proj_decode(sp_plan_t plan, const void* spikes, sp_fmt fmt, int32_t* acc, float* y,
                            sp_stream_t stream) {
  if (!plan) return SP_EINVAL;
  sp_status st = check_io(spikes, fmt, acc, y);
  if (st != SP_OK) return st;
  return run_gather(plan, spikes, fmt, 1, row_elems(fmt, plan->K), acc, y, as_stream(stream));
}

sp_status spike_proj_batched(sp_plan_t plan, const void* spikes, sp_fmt fmt, int32_t B,
                             int64_t ld_spikes, int32_t* acc, float* y, sp_kernel strategy,
                             sp_stream_t stream) {
  if (!plan) return SP_EINVAL;
  sp_status st = check_io(spikes, fmt, acc, y);
  if (st != SP_OK) return st;
  if (B < 1) return SP_EINVAL;
  if (B > plan->max_batch) return SP_ERANGE;
  if (ld_spikes < row_elems(fmt, plan->K)) return SP_EINVAL;
  if (strategy < SP_AUTO || strategy > SP_GEMM) return SP_EINVAL;
  if (strategy == SP_GEMM && !(plan->flags & SP_PLAN_GEMM)) return SP_EUNSUPPORTED;
  return run_multi(plan, spikes, fmt, B, ld_spikes, acc, y, strategy, as_stream(stream));
}

sp_status spike_proj_prefill(sp_plan_t plan, const uint8_t* X, int32_t T, int64_t ldx,
                             int32_t* acc, float* y, sp_kernel strategy, sp_stream_t stream) {
  return spike_proj_batched(plan, X, SP_SPIKES_U8, T, ldx, acc, y, strategy, stream);
}

sp_status spike_proj_last_dispatch(sp_plan_t plan, sp_kernel* chosen, int32_t* active_count) {
  if (!plan) return SP_EINVAL;
  if (chosen) *chosen = plan->last_kernel;
  if (active_count) *active_count = plan->last_active;
  return SP_OK;
}

sp_status spike_proj_plan_status(sp_plan_t plan, sp_stream_t stream) {
  if (!plan) return SP_EINVAL;
  cudaStream_t s = as_stream(stream);
  int h = 0;
  SP_CUDA(cudaMemcpyAsync(&h, plan->err, sizeof(int), cudaMemcpyDeviceToHost, s));
  SP_CUDA(cudaStreamSynchronize(s));
  if (h == 0) return SP_OK;
  SP_CUDA(cudaMemsetAsync(plan->err, 0, sizeof(int), s));
  SP_CUDA(cudaMemsetAsync(plan->ws, 0, (size_t)plan->max_batch * plan->N * sizeof(int32_t), s));
  SP_CUDA(cudaMemsetAsync(plan->tickets, 0, plan->n_tickets * sizeof(uint32_t), s));
  SP_CUDA(cudaStreamSynchronize(s));
  return SP_EKERNEL;
}

// ---------------------------------------------------------------------------
sp_status spike_proj_group_create(sp_group_t* group, const sp_plan_t* plans, int32_t count,
                                  sp_stream_t stream) {
  if (!group || !plans || count < 1 || count > SPIKE_PROJ_MAX_GROUP) return SP_EINVAL;
  int dev = 0;
  sp_status st = check_device(&dev);
  if (st != SP_OK) return st;
  for (int j = 0; j < count; ++j)
    if (!plans[j] || plans[j]->device != dev) return SP_EINVAL;
  cudaStream_t s = as_stream(stream);
  sp_group_s* g = new (std::nothrow) sp_group_s();
  if (!g) return SP_ENOMEM;
  g->count = count;
  std::memset(&g->params, 0, sizeof(g->params));
  int64_t units = 0, ws = 0, tk = 0;
  for (int j = 0; j < count; ++j) {
    sp_plan_s* p = plans[j];
    g->plans[j] = p;
    GatherProblem& P = g->params.prob[j];
    P.W = p->W;
    P.scale = p->scale;
    P.ldw = (int32_t)p->ldw;
    P.N = p->N;
    P.K = p->K;
    P.unit_begin = (int32_t)units;
    P.ws_begin = (int32_t)ws;
    P.ticket_begin = (int32_t)tk;
    units += gather_units(p->N, p->K);
    if (gather_units(p->N, p->K) > g->params.max_units) g->params.max_units = gather_units(p->N, p->K);
    ws += p->N;
    tk += gather_ntiles(p->N);
    if (p->N > g->maxN) g->maxN = p->N;
    if (p->K > g->maxK) g->maxK = p->K;
  }
  if (units > INT32_MAX || ws > INT32_MAX) {
    delete g;
    return SP_ERANGE;
  }
  g->params.nprob = count;
  g->params.B = 1;
  g->params.units_total = (int32_t)units;
  g->ws_elems = (size_t)ws;
  g->n_tickets = (size_t)tk;
  g->spike_row_bytes = (size_t)g->maxK;   // covers both formats (ceil(K/32)*4 <= K+3)
  g->spike_row_bytes = (g->spike_row_bytes + 15) / 16 * 16;
  if ((st = dev_alloc_zero(&g->ws, g->ws_elems, s)) != SP_OK ||
      (st = dev_alloc_zero(&g->tickets, g->n_tickets, s)) != SP_OK ||
      (st = dev_alloc_zero(&g->err, 1, s)) != SP_OK ||
      (st = dev_alloc_zero(reinterpret_cast<uint8_t**>(&g->d_spikes),
                           (size_t)count * g->spike_row_bytes, s)) != SP_OK ||
      (st = dev_alloc_zero(&g->d_acc, (size_t)count * g->maxN, s)) != SP_OK ||
      (st = dev_alloc_zero(&g->d_y, (size_t)count * g->maxN, s)) != SP_OK) {
    group_free(g);
    return st;
  }
  bool all_gemm = true;
  for (int j = 0; j < count; ++j) all_gemm = all_gemm && (plans[j]->flags & SP_PLAN_GEMM);
  if (all_gemm &&
      ((st = dev_alloc_zero(&g->gpart, (size_t)kGemmGroupSlots * kGemmPartialElems, s)) != SP_OK ||
       (st = dev_alloc_zero(&g->gflags, (size_t)kGemmGroupSlots * 8, s)) != SP_OK)) {
    group_free(g);
    return st;
  }
  g->params.ws = g->ws;
  g->params.tickets = g->tickets;
  g->params.err = g->err;
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    group_free(g);
    return cuda_fail(e);
  }
  *group = g;
  return SP_OK;
}

sp_status spike_proj_group_destroy(sp_group_t group) {
  if (!group) return SP_OK;
  cudaError_t e = cudaDeviceSynchronize();
  group_free(group);
  return e == cudaSuccess ? SP_OK : cuda_fail(e);
}

sp_status spike_proj_group_decode(sp_group_t g, const void* spikes, sp_fmt fmt, int64_t ld_spikes,
                                  int32_t* acc, float* y, int64_t ld_out, sp_stream_t stream) {
  if (!g) return SP_EINVAL;
  sp_status st = check_io(spikes, fmt, acc, y);
  if (st != SP_OK) return st;
  if (ld_spikes < row_elems(fmt, g->maxK) || ld_out < g->maxN) return SP_EINVAL;
  GatherParamsG& P = g->params;
  P.fmt = fmt;
  P.spikes = spikes;
  P.ld_spikes = ld_spikes;
  P.acc = acc;
  P.y = y;
  P.ld_out = ld_out;
  P.fault = g->fault;
  g->fault = 0;
  const cudaError_t e = launch_gather(P, as_stream(stream));
  P.fault = 0;
  SP_CUDA(e);
  return SP_OK;
}

sp_status spike_proj_group_prefill(sp_group_t g, const void* const* X, sp_fmt fmt, int32_t T,
                                   int64_t ldx, int32_t* const* acc, float* const* y,
                                   sp_stream_t stream) {
  if (!g || !X || !fmt_ok(fmt) || T < 1 || (!acc && !y)) return SP_EINVAL;
  for (int j = 0; j < g->count; ++j) {
    const sp_plan_s* p = g->plans[j];
    if (!(p->flags & SP_PLAN_GEMM)) return SP_EUNSUPPORTED;
    if (T > p->max_batch) return SP_ERANGE;
    if (!X[j] || (acc && !acc[j]) || (y && !y[j])) return SP_EINVAL;
    if (ldx < row_elems(fmt, p->K)) return SP_EINVAL;
    if (fmt == SP_SPIKES_BITS32 && !aligned(X[j], 4)) return SP_EALIGN;
    if ((acc && !aligned(acc[j], 4)) || (y && !aligned(y[j], 4))) return SP_EALIGN;
  }
  if (!g->gemm) {
    g->gemm = new (std::nothrow) GemmGroupArgs();
    if (!g->gemm) return SP_ENOMEM;
  }
  cudaStream_t s = as_stream(stream);
  GemmGroupArgs& a = *g->gemm;
  a.count = g->count;
  a.err = g->err;
  a.part = g->gpart;
  a.flags = g->gflags;
  int64_t units = 0;
  // CTA pairs (2-SM MMA over 256 rows) when the members' row tiles pair up
  // with little padding
  int tm[kMaxProblems], tn[kMaxProblems];
  for (int j = 0; j < g->count; ++j) {
    tm[j] = ceil_div(T, 128);
    tn[j] = ceil_div(g->plans[j]->N, 256);
  }
  const int cl = gemm_group_cluster(tm, tn, g->count);
  a.cl = cl;
  // 0/1 byte rows that TMA can address are read in place; any other input
  // is first written as 0/1 bytes into the member plan's staging copy
  const bool vec = fmt == SP_SPIKES_BOOL8 && ldx % 16 == 0;
  for (int j = 0; j < g->count; ++j) {
    sp_plan_s* p = g->plans[j];
    GemmMember& M = a.m[j];
    if (vec && aligned(X[j], 16)) {
      if (X[j] != g->rows_ptr[j] || ldx != g->rows_ld[j] || T != g->rows_T[j]) {
        SP_CUDA(gemm_make_rows_map(X[j], ldx, T, p->K, &g->rows_map[j]));
        g->rows_ptr[j] = X[j];
        g->rows_ld[j] = ldx;
        g->rows_T[j] = T;
      }
      M.a = g->rows_map[j];
    } else {
      SP_CUDA(launch_spikes_to_01(X[j], fmt, ldx, T, p->K, p->Kp, p->Xs, s));
      M.a = p->maps.a;
    }
    M.b = cl == 2 ? p->maps.b128 : p->maps.b;
    M.p.scale = p->scale;
    M.p.acc = acc ? acc[j] : nullptr;
    M.p.y = y ? y[j] : nullptr;
    M.p.T = T;
    M.p.N = p->N;
    M.p.K = p->K;
    M.p.err = g->err;
    M.p.part = nullptr;
    M.p.part_units = 0;
    M.p.fault = g->fault;
    M.tiles_n = tn[j];
    M.nkb = p->Kp / 64;
    M.unit_begin = (int32_t)units;
    units += (int64_t)ceil_div(tm[j], cl) * tn[j];
    if (units > INT32_MAX) return SP_ERANGE;
    M.unit_end = (int32_t)units;
  }
  a.units = (int32_t)units;
  g->fault = 0;
  SP_CUDA(launch_gemm_group(a, s));
  return SP_OK;
}

sp_status spike_proj_group_decode_host(sp_group_t g, const void* h_spikes, sp_fmt fmt,
                                       int64_t ld_spikes, int32_t* h_acc, float* h_y,
                                       int64_t ld_out, sp_stream_t stream) {
  if (!g || !h_spikes || !fmt_ok(fmt) || (!h_acc && !h_y)) return SP_EINVAL;
  const int64_t need = row_elems(fmt, g->maxK);
  if (ld_spikes < need || ld_out < g->maxN) return SP_EINVAL;
  if ((fmt == SP_SPIKES_BITS32 && !aligned(h_spikes, 4)) || (h_acc && !aligned(h_acc, 4)) ||
      (h_y && !aligned(h_y, 4)))
    return SP_EALIGN;
  cudaStream_t s = as_stream(stream);
  const size_t elem = fmt == SP_SPIKES_BITS32 ? 4 : 1;
  const size_t row_bytes = (size_t)need * elem;
  GatherParamsG& P = g->params;
  P.fmt = fmt;
  // Page-locked host buffers are read and written by the kernel in place;
  // pageable ones go through the group's device staging.
  const void* m_spikes = device_view(h_spikes);
  if (m_spikes) {
    P.spikes = m_spikes;
    P.ld_spikes = ld_spikes;
  } else {
    SP_CUDA(cudaMemcpy2DAsync(g->d_spikes, g->spike_row_bytes, h_spikes, (size_t)ld_spikes * elem,
                              row_bytes, (size_t)g->count, cudaMemcpyHostToDevice, s));
    P.spikes = g->d_spikes;
    P.ld_spikes = (int64_t)(g->spike_row_bytes / elem);
  }
  int32_t* m_acc = h_acc ? static_cast<int32_t*>(device_view(h_acc)) : nullptr;
  float* m_y = h_y ? static_cast<float*>(device_view(h_y)) : nullptr;
  const bool out_mapped = (!h_acc || m_acc) && (!h_y || m_y);
  if (out_mapped) {
    P.acc = m_acc;
    P.y = m_y;
    P.ld_out = ld_out;
  } else {
    P.acc = h_acc ? g->d_acc : nullptr;
    P.y = h_y ? g->d_y : nullptr;
    P.ld_out = g->maxN;
  }
  P.fault = g->fault;
  g->fault = 0;
  const cudaError_t el = launch_gather(P, s);
  P.fault = 0;
  SP_CUDA(el);
  if (out_mapped) return SP_OK;
  const size_t out_row = (size_t)g->maxN * 4;
  if (h_acc)
    SP_CUDA(cudaMemcpy2DAsync(h_acc, (size_t)ld_out * 4, g->d_acc, out_row, out_row,
                              (size_t)g->count, cudaMemcpyDeviceToHost, s));
  if (h_y)
    SP_CUDA(cudaMemcpy2DAsync(h_y, (size_t)ld_out * 4, g->d_y, out_row, out_row, (size_t)g->count,
                              cudaMemcpyDeviceToHost, s));
  return SP_OK;
}

namespace {
// true when the byte ranges [a, a + na) and [b, b + nb) share a byte
bool overlaps(const void* a, int64_t na, const void* b, int64_t nb) {
  const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
  return x < y + (uintptr_t)nb && y < x + (uintptr_t)na;
}
}  // namespace

sp_status spike_proj_group_decode_lif(sp_group_t g, const float* v_in, float* v_out,
                                      const float* I, int64_t ld, float beta, float theta,
                                      uint32_t* bits, int64_t ld_bits, int32_t* acc, float* y,
                                      int64_t ld_out, sp_stream_t stream) {
  if (!g || !v_in || !v_out || !I || (!acc && !y)) return SP_EINVAL;
  if (ld < g->maxK || ld_out < g->maxN || (bits && ld_bits < words_for(g->maxK))) return SP_EINVAL;
  if (!aligned(v_in, 4) || !aligned(v_out, 4) || !aligned(I, 4) || (bits && !aligned(bits, 4)) ||
      (acc && !aligned(acc, 4)) || (y && !aligned(y, 4)))
    return SP_EALIGN;
  const int64_t state_bytes = ((int64_t)(g->count - 1) * ld + g->maxK) * 4;
  const int64_t bits_bytes = bits ? ((int64_t)(g->count - 1) * ld_bits + words_for(g->maxK)) * 4 : 0;
  if (overlaps(v_out, state_bytes, v_in, state_bytes) || overlaps(v_out, state_bytes, I, state_bytes))
    return SP_EINVAL;
  if (bits && (overlaps(bits, bits_bytes, v_in, state_bytes) ||
               overlaps(bits, bits_bytes, v_out, state_bytes) ||
               overlaps(bits, bits_bytes, I, state_bytes)))
    return SP_EINVAL;
  cudaStream_t s = as_stream(stream);
  GatherParamsG q = g->params;
  q.acc = acc;
  q.y = y;
  q.ld_out = ld_out;
  q.fmt = SP_SPIKES_BITS32;
  q.lif_vin = v_in;
  q.lif_vout = v_out;
  q.lif_I = I;
  q.lif_ld = ld;
  q.lif_beta = beta;
  q.lif_theta = theta;
  q.lif_bits = bits;
  q.lif_ld_bits = ld_bits;
  q.spikes = nullptr;
  q.ld_spikes = 0;
  q.fault = g->fault;
  g->fault = 0;
  const cudaError_t e = launch_gather(q, s);
  if (e != cudaErrorNotSupported) {
    SP_CUDA(e);
    return SP_OK;
  }
  // the fused form does not apply: the producer into bits (or the group's
  // staging rows), then the decode of those rows
  uint32_t* b = bits ? bits : static_cast<uint32_t*>(g->d_spikes);
  const int64_t ldb = bits ? ld_bits : (int64_t)(g->spike_row_bytes / 4);
  int32_t Ks[kMaxProblems];
  for (int j = 0; j < g->count; ++j) Ks[j] = q.prob[j].K;
  SP_CUDA(launch_lif_rows(v_in, v_out, I, Ks, g->count, ld, beta, theta, b, ldb, s));
  q.lif_vin = nullptr;
  q.lif_vout = nullptr;
  q.lif_I = nullptr;
  q.lif_bits = nullptr;
  q.spikes = b;
  q.ld_spikes = ldb;
  SP_CUDA(launch_gather(q, s));
  return SP_OK;
}

sp_status spike_proj_group_status(sp_group_t g, sp_stream_t stream) {
  if (!g) return SP_EINVAL;
  cudaStream_t s = as_stream(stream);
  int h = 0;
  SP_CUDA(cudaMemcpyAsync(&h, g->err, sizeof(int), cudaMemcpyDeviceToHost, s));
  SP_CUDA(cudaStreamSynchronize(s));
  if (h == 0) return SP_OK;
  SP_CUDA(cudaMemsetAsync(g->err, 0, sizeof(int), s));
  SP_CUDA(cudaMemsetAsync(g->ws, 0, g->ws_elems * sizeof(int32_t), s));
  SP_CUDA(cudaMemsetAsync(g->tickets, 0, g->n_tickets * sizeof(uint32_t), s));
  if (g->gflags)
    SP_CUDA(cudaMemsetAsync(g->gflags, 0, (size_t)kGemmGroupSlots * 8 * sizeof(uint32_t), s));
  SP_CUDA(cudaStreamSynchronize(s));
  return SP_EKERNEL;
}

sp_status spike_proj_decode_noalloc(const int8_t* W, int64_t ldw, const float* scale, int32_t N,
                                    int32_t K, const void* spikes, sp_fmt fmt, int32_t* acc,
                                    float* y, sp_stream_t stream) {
  if (!W || !scale) return SP_EINVAL;
  sp_status st = check_io(spikes, fmt, acc, y);
  if (st != SP_OK) return st;
  if (N < 16) return SP_EINVAL;
  if (N > kNoallocMaxN) return SP_ESCRATCH;
  if (K < 1 || K > SPIKE_PROJ_MAX_K) return SP_ERANGE;
  if (N % 16 != 0 || ldw < N || ldw % 16 != 0 || ldw > INT32_MAX) return SP_EALIGN;
  if (!aligned(W, 16) || !aligned(scale, 4)) return SP_EALIGN;
  cudaStream_t s = as_stream(stream);
  int32_t* scratch = nullptr;
  if ((st = noalloc_scratch(s, &scratch)) != SP_OK) return st;
  GatherParams1 g;
  std::memset(&g, 0, sizeof(g));
  g.prob[0].W = W;
  g.prob[0].scale = scale;
  g.prob[0].ldw = (int32_t)ldw;
  g.prob[0].N = N;
  g.prob[0].K = K;
  g.nprob = 1;
  g.B = 1;
  g.units_total = gather_units(N, K);
  g.max_units = gather_units(N, K);
  g.fmt = fmt;
  g.spikes = spikes;
  g.ld_spikes = row_elems(fmt, K);
  g.acc = acc;
  g.y = y;
  g.ld_out = N;
  g.ws = scratch;
  g.tickets = reinterpret_cast<uint32_t*>(scratch + kNoallocMaxN);
  g.err = nullptr;                        // no status word: see the header
  SP_CUDA(launch_gather(g, s));
  return SP_OK;
}

sp_status spike_proj_plan_inject_fault(sp_plan_t plan, int32_t fault) {
  if (!plan || fault < SP_FAULT_NONE || fault > SP_FAULT_STALL) return SP_EINVAL;
  plan->fault = fault;
  return SP_OK;
}

sp_status spike_proj_group_inject_fault(sp_group_t group, int32_t fault) {
  if (!group || fault < SP_FAULT_NONE || fault > SP_FAULT_STALL) return SP_EINVAL;
  group->fault = fault;
  return SP_OK;
}

sp_status spike_proj_probe_gather(const void* base, const uint32_t* offsets16, int32_t count,
                                  int32_t piece_bytes, uint32_t* sink, sp_stream_t stream) {
  if (!base || !sink || count < 0 || (count > 0 && !offsets16)) return SP_EINVAL;
  if (piece_bytes != 512 && piece_bytes != 1024 && piece_bytes != 1536) return SP_EINVAL;
  if (!aligned(base, 16) || !aligned(sink, 4) || (offsets16 && !aligned(offsets16, 4)))
    return SP_EALIGN;
  int dev = 0;
  const sp_status st = check_device(&dev);
  if (st != SP_OK) return st;
  SP_CUDA(launch_probe_gather(static_cast<const uint8_t*>(base), offsets16, count, piece_bytes,
                              sink, as_stream(stream)));
  return SP_OK;
}

sp_status spike_proj_lif(float* v, const float* I, int32_t K, int32_t rows, int64_t ld,
                         float beta, float theta, uint32_t* bits, int64_t ld_bits,
                         sp_stream_t stream) {
  if (!v || !I || !bits || rows < 1 || K < 1) return SP_EINVAL;
  if (K > SPIKE_PROJ_MAX_K) return SP_ERANGE;
  if (ld < K || ld_bits < words_for(K)) return SP_EINVAL;
  if (!aligned(v, 4) || !aligned(I, 4) || !aligned(bits, 4)) return SP_EALIGN;
  int dev = 0;
  const sp_status st = check_device(&dev);
  if (st != SP_OK) return st;
  SP_CUDA(launch_lif(v, I, K, rows, ld, beta, theta, bits, ld_bits, as_stream(stream)));
  return SP_OK;
}

sp_status spike_proj_dense(const sp_dense* problems, int32_t count, int32_t B,
                           sp_stream_t stream) {
  if (!problems || count < 1 || count > SPIKE_PROJ_DENSE_MAX_GROUP || B < 1 ||
      B > SPIKE_PROJ_DENSE_MAX_B)
    return SP_EINVAL;
  DenseProblem probs[kDenseMaxProblems];
  for (int j = 0; j < count; ++j) {
    const sp_dense& d = problems[j];
    if (!d.W || !d.scale || !d.x || !d.y || d.N < 1 || d.K < 1 || d.ldy < d.N) return SP_EINVAL;
    if (d.K > SPIKE_PROJ_MAX_K) return SP_ERANGE;
    if (d.ldw < d.K || d.ldw % 16 != 0 || !aligned(d.W, 16)) return SP_EALIGN;
    if (d.ldx < d.K || d.ldx % 4 != 0 || !aligned(d.x, 16)) return SP_EALIGN;
    if (!aligned(d.scale, 4) || !aligned(d.y, 4)) return SP_EALIGN;
    probs[j] = DenseProblem{d.W, d.ldw, d.scale, d.x, d.ldx, d.y, d.ldy, d.N, d.K};
  }
  int dev = 0;
  const sp_status st = check_device(&dev);
  if (st != SP_OK) return st;
  SP_CUDA(launch_dense(probs, count, B, as_stream(stream)));
  return SP_OK;
}

// ---------------------------------------------------------------------------
sp_status spike_proj_head_create(sp_head_t* head, const int8_t* W, int64_t ldw, const float* scale,
                                 int32_t V, int32_t K, sp_stream_t stream) {
  if (!head || !W || !scale) return SP_EINVAL;
  if (V < 2 || V > SPIKE_PROJ_HEAD_MAX_V || K < 1 || K > SPIKE_PROJ_HEAD_MAX_K) return SP_ERANGE;
  if (ldw < K || ldw % 16 != 0 || !aligned(W, 16) || !aligned(scale, 4)) return SP_EALIGN;
  int dev = 0;
  sp_status st = check_device(&dev);
  if (st != SP_OK) return st;
  cudaStream_t s = as_stream(stream);
  sp_head_s* hd = new (std::nothrow) sp_head_s();
  if (!hd) return SP_ENOMEM;
  hd->device = dev;
  hd->W = W;
  hd->ldw = ldw;
  hd->scale = scale;
  hd->V = V;
  hd->K = K;
  if ((st = dev_alloc_zero(&hd->ws, head_workspace_bytes(), s)) != SP_OK) {
    delete hd;
    return st;
  }
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    cudaFree(hd->ws);
    delete hd;
    return cuda_fail(e);
  }
  *head = hd;
  return SP_OK;
}

sp_status spike_proj_head_destroy(sp_head_t head) {
  if (!head) return SP_OK;
  cudaError_t e = cudaDeviceSynchronize();
  cudaFree(head->ws);
  delete head;
  return e == cudaSuccess ? SP_OK : cuda_fail(e);
}

sp_status spike_proj_head(sp_head_t hd, const float* h, int64_t ldh, int32_t B, float tau,
                          int32_t k_sel, int32_t* token, int32_t* verified, float* gap,
                          int32_t* cand, float* r, float* z, int64_t ld_z, sp_stream_t stream) {
  if (!hd || !h || !token || B < 1 || B > SPIKE_PROJ_HEAD_MAX_B) return SP_EINVAL;
  if (k_sel < 1 || k_sel > SPIKE_PROJ_HEAD_MAX_CAND || k_sel > hd->V) return SP_EINVAL;
  if (ldh < hd->K || (z && ld_z < hd->V)) return SP_EINVAL;
  if (!aligned(h, 16) || ldh % 4 != 0) return SP_EALIGN;
  if (!aligned(token, 4) || (verified && !aligned(verified, 4)) || (gap && !aligned(gap, 4)) ||
      (cand && !aligned(cand, 4)) || (r && !aligned(r, 4)) || (z && !aligned(z, 4)))
    return SP_EALIGN;
  HeadArgs a;
  a.W = hd->W;
  a.ldw = hd->ldw;
  a.scale = hd->scale;
  a.V = hd->V;
  a.K = hd->K;
  a.h = h;
  a.ldh = ldh;
  a.B = B;
  a.tau = tau;
  a.k_sel = k_sel;
  a.token = token;
  a.verified = verified;
  a.gap = gap;
  a.cand = cand;
  a.r = r;
  a.z = z;
  a.ld_z = ld_z;
  a.ws = hd->ws;
  SP_CUDA(launch_head(a, as_stream(stream)));
  return SP_OK;
}

const char* spike_proj_strerror(sp_status status) {
  switch (status) {
    case SP_OK: return "success";
    case SP_EINVAL: return "invalid argument";
    case SP_EALIGN: return "alignment or leading-dimension rule violated";
    case SP_EDEVICE: return "current device is not compute capability 10.3 (GB300)";
    case SP_ECUDA: return "CUDA runtime error (see spike_proj_last_cuda_error)";
    case SP_ENOMEM: return "device memory allocation failed";
    case SP_ERANGE: return "size out of range (K above 131072 or batch above the plan's maximum)";
    case SP_EKERNEL: return "a kernel reported an error (device error word set)";
    case SP_EUNSUPPORTED: return "strategy not available for this plan";
    case SP_ESCRATCH:
      return "N above SPIKE_PROJ_NOALLOC_MAX_N (32768): too large for the fixed scratch of "
             "spike_proj_decode_noalloc";
  }
  return "unknown status";
}

int spike_proj_last_cuda_error(void) { return g_last_cuda_error; }
int spike_proj_abi_version(void) { return SPIKE_PROJ_ABI_VERSION; }

}  // extern "C"
