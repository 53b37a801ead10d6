// Routing by ancestry in front of replicated aggregators (Alto, arxiv
// 2403.04311, Sec. 4.3: every element with the same ancestry tags goes to the
// same instance, a new flow may be placed by load; Sec. 5: replicas chosen by
// routing rules and queue lengths), on one GB300.
//
// One batch (stream-ordered, no host synchronisation):
//   begin    batch counters
//   assign   per fragment: check its payload offsets; its flow is the group at
//            the routing level; HASH: splitmix64 of the flow key mod R;
//            LEAST_LOADED: find or insert the flow in the flow table, and for
//            a flow not yet placed note its first fragment (atomicMin)
//   rank     (LEAST_LOADED) look-back scan: new flows numbered in the order
//            of their first fragment
//   order    one CTA: replicas ranked by load at the batch start
//   place    (LEAST_LOADED) each new flow takes order[rank mod R]
//   final    per fragment: its replica, per-replica counts
//   offsets  one CTA: replica fragment offsets; loads += counts
//   sort     stable onesweep radix sort of the fragments by replica
//   lengths  look-back scan of payload lengths in replica order
//   scatter  per fragment: tags into the replica's level-major block, its
//            payload offset, its score
//   copy     payload spans, eight lanes a span (as the aggregator's gather)
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <new>
#include <vector>

#include "alto_agg.h"
#include "common.cuh"
#include "kernels.h"
#include "scan.cuh"

namespace alto {
namespace {

constexpr int kRT = 256;

struct RDev {
  Ctl* ctl;
  int depth, level, R, policy, with_score;
  u32 nmax;
  u64 max_pay;
  // flow table (LEAST_LOADED): a slot's replica and first fragment are kNone
  // whenever the slot is free, so an insert writes only the key
  u64* fkey;
  u32* frep;
  u32* ffirst;
  u32 fmask;
  int fprobe;
  u32* freed;      // [nmax] slots released by the last release call
  // the batch
  const u64* tags;
  const u32* off;
  const int32_t* pay;
  const float* score;
  u32 n;
  u64 n_payload;
  // scratch and state
  u32* fe;         // [nmax] flow slot of each fragment
  u32* rank;       // [nmax] number of new flows first seen before each fragment
  u32* order;      // [R] replicas by load at the batch start
  u64* load;       // [R] fragments routed to each replica so far
  u32* counts;     // [R] fragments of this batch per replica
  u32* rep_key;    // [nmax] replica of each fragment (the sort's input keys)
  // outputs
  u32* replica;    // [nmax]
  const u32* perm;
  const u32* skey;
  int64_t* frag_off;  // [R + 1]
  int64_t* pay_off;   // [R + 1]
  u64* ppos;          // [nmax + 1] payload position of each fragment in replica order
  u64* out_tags;      // [depth * nmax]
  u32* out_poff;      // [nmax + R]
  int32_t* out_pay;   // [max_pay]
  float* out_score;   // [nmax]
};

__device__ __forceinline__ u64 flow_key(const RDev& d, u32 i) {
  return ((u64)d.level << 32) | tag_pid(d.tags[(u64)d.level * d.n + i]);
}

__global__ void k_rt_begin(RDev d, u32 n) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (threadIdx.x == 0) {
    ctl->epoch += 1;
    ctl->batch_err = 0;
    ctl->n = (ctl->status == ALTO_OK) ? n : 0u;
    ctl->n_done = 0;
  }
  for (int r = threadIdx.x; r < d.R; r += blockDim.x) d.counts[r] = 0;
}

// The flow's slot, inserted if new.  A walk from the home slot ends at the
// key or at the first free slot; a new key takes the first released slot
// (tombstone) it passed, else that free slot, so that released flows do not
// fill the table.  Slots only go from free or released to a key within a
// launch: a lost compare-and-swap means another key took the slot, and the
// walk goes on from there; a key lies within fprobe slots of home.
__device__ u32 flow_find_or_insert(const RDev& d, u64 key) {
  const u32 home = (u32)mix64(key) & d.fmask;
  const u32 reach = (u32)d.fprobe;  // at most the table size
  u32 h = home, dist = 0;
  u32 tomb_at = kNone;
  for (;;) {
    if (dist < reach) {
      const u64 cur = ((volatile u64*)d.fkey)[h];
      if (cur == key) return h;
      if (cur == kTomb && tomb_at == kNone) tomb_at = h;
      if (cur != kEmpty) {
        h = (h + 1) & d.fmask;
        ++dist;
        continue;
      }
    } else if (tomb_at == kNone) {
      break;
    }
    const u32 t = (tomb_at != kNone) ? tomb_at : h;
    const u64 want = (tomb_at != kNone) ? kTomb : kEmpty;
    const u64 prev = atomicCAS((unsigned long long*)&d.fkey[t], (unsigned long long)want,
                               (unsigned long long)key);
    if (prev == want || prev == key) return t;
    h = t;  // its distance from home is below reach: no wrap
    dist = (t - home) & d.fmask;
    tomb_at = kNone;
  }
  raise_err(d.ctl, ALTO_ENOSPC);
  return kNone;
}

__global__ void __launch_bounds__(kRT) k_rt_assign(RDev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (halted(ctl)) return;
  const u32 n = ctl->n;
  for (u32 i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    const u32 o0 = d.off[i], o1 = d.off[i + 1];
    if (o1 < o0 || (u64)o1 > d.n_payload) raise_err(ctl, ALTO_EINVAL);
    const u64 key = flow_key(d, i);
    if (d.policy == ALTO_ROUTE_HASH) {
      d.rep_key[i] = (u32)(mix64(key) % (u64)d.R);
      continue;
    }
    const u32 e = flow_find_or_insert(d, key);
    d.fe[i] = e;
    if (e != kNone && d.frep[e] == kNone) atomicMin(&d.ffirst[e], i);
  }
}

// New flows numbered in the order of their first fragment.
struct RankScan2 {
  RDev d;
  __device__ u64 size(const Ctl* ctl) const { return ctl->n; }
  __device__ u64 value(u64 i) const {
    const u32 e = d.fe[i];
    return (e != kNone && d.frep[e] == kNone && d.ffirst[e] == (u32)i) ? 1u : 0u;
  }
  __device__ void out(u64 i, u64 excl, u64) const { d.rank[i] = (u32)excl; }
  __device__ void total(Ctl* ctl, u64 t) const { ctl->n_done = (u32)t; }
};

// One CTA: replica r goes to position #{r' : (load r', r') < (load r, r)}.
__global__ void __launch_bounds__(1024) k_rt_order(RDev d) {
  pdl_enter();
  for (int r = threadIdx.x; r < d.R; r += blockDim.x) {
    const u64 lr = d.load[r];
    int pos = 0;
    for (int q = 0; q < d.R; ++q) {
      const u64 lq = d.load[q];
      pos += (lq < lr || (lq == lr && q < r)) ? 1 : 0;
    }
    d.order[pos] = (u32)r;
  }
}

__global__ void __launch_bounds__(kRT) k_rt_place(RDev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (halted(ctl)) return;
  const u32 n = ctl->n;
  for (u32 i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    const u32 e = d.fe[i];
    if (e == kNone || d.frep[e] != kNone || d.ffirst[e] != i) continue;
    d.frep[e] = d.order[d.rank[i] % (u32)d.R];
    d.ffirst[e] = kNone;
  }
}

__global__ void __launch_bounds__(kRT) k_rt_final(RDev d) {
  pdl_enter();
  __shared__ u32 s_cnt[ALTO_MAX_REPLICAS];
  Ctl* ctl = d.ctl;
  for (int r = threadIdx.x; r < d.R; r += blockDim.x) s_cnt[r] = 0;
  __syncthreads();
  const u32 n = halted(ctl) ? 0 : ctl->n;
  for (u32 i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    u32 r;
    if (d.policy == ALTO_ROUTE_HASH) {
      r = d.rep_key[i];
    } else {
      const u32 e = d.fe[i];
      r = (e == kNone) ? 0u : d.frep[e];
      if (r >= (u32)d.R) r = 0;  // only after an error (a full flow table)
      d.rep_key[i] = r;
    }
    d.replica[i] = r;
    atomicAdd(&s_cnt[r], 1u);
  }
  __syncthreads();
  for (int r = threadIdx.x; r < d.R; r += blockDim.x)
    if (s_cnt[r]) atomicAdd(&d.counts[r], s_cnt[r]);
}

// One CTA of 1024: replica fragment offsets (a block scan) and the new loads.
__global__ void __launch_bounds__(1024) k_rt_offsets(RDev d) {
  pdl_enter();
  __shared__ u64 s_w[32];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const u64 c = (t < d.R) ? d.counts[t] : 0u;
  u64 x = c;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const u64 y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s_w[warp] = x;
  __syncthreads();
  u64 pre = 0;
  for (int q = 0; q < warp; ++q) pre += s_w[q];
  if (t < d.R) {
    d.frag_off[t] = (int64_t)(pre + x - c);
    d.load[t] += c;
  }
  if (t == d.R - 1) d.frag_off[d.R] = (int64_t)(pre + x);
}

__global__ void __launch_bounds__(kRT) k_rt_identity(RDev d, u32* perm) {
  pdl_enter();
  const u32 n = d.ctl->n;
  for (u32 j = blockIdx.x * blockDim.x + threadIdx.x; j < n; j += gridDim.x * blockDim.x) perm[j] = j;
}

// Payload lengths in replica order.
struct PermLenScan {
  RDev d;
  __device__ u64 size(const Ctl* ctl) const { return ctl->batch_err ? 0 : ctl->n; }
  __device__ u64 value(u64 j) const {
    const u32 i = d.perm[j];
    return d.off[i + 1] - d.off[i];
  }
  __device__ void out(u64 j, u64 excl, u64) const { d.ppos[j] = excl; }
  __device__ void total(Ctl* ctl, u64 t) const { d.ppos[size(ctl)] = t; }
};

__global__ void __launch_bounds__(kRT) k_rt_scatter(RDev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (halted(ctl) || ctl->batch_err) return;
  const u32 n = ctl->n;
  const u32 g = blockIdx.x * blockDim.x + threadIdx.x, stride = gridDim.x * blockDim.x;
  for (u32 r = g; r <= (u32)d.R; r += stride) {
    const int64_t fo = d.frag_off[r];
    d.pay_off[r] = (int64_t)d.ppos[fo];
    if (r < (u32)d.R && d.frag_off[r + 1] == fo) d.out_poff[fo + r] = 0;  // an empty sub-batch
  }
  for (u32 j = g; j < n; j += stride) {
    const u32 i = d.perm[j];
    const u32 r = (d.R > 1) ? d.skey[j] : 0u;
    const u64 fo = (u64)d.frag_off[r], nr = (u64)d.frag_off[r + 1] - fo, q = j - fo;
    for (int l = 0; l < d.depth; ++l) d.out_tags[(u64)d.depth * fo + (u64)l * nr + q] = d.tags[(u64)l * n + i];
    const u64 pb = d.ppos[fo];
    d.out_poff[fo + r + q] = (u32)(d.ppos[j] - pb);
    if (q + 1 == nr) d.out_poff[fo + r + nr] = (u32)(d.ppos[j + 1] - pb);
    if (d.with_score) d.out_score[j] = d.score[i];
  }
}

// Payload spans in replica order: eight lanes a span, loads before stores.
__global__ void __launch_bounds__(kRT) k_rt_copy(RDev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (halted(ctl) || ctl->batch_err) return;
  const u32 n = ctl->n;
  const int lane = threadIdx.x & 31, sub = lane & 7, grp = lane >> 3;
  const u64 gw = (blockIdx.x * (u64)blockDim.x + threadIdx.x) >> 5, nw = (gridDim.x * (u64)blockDim.x) >> 5;
  for (u64 jb = gw * 4; jb < n; jb += nw * 4) {
    const u64 j = jb + grp;
    u32 len = 0;
    const int32_t* src = d.pay;
    int32_t* dst = d.out_pay;
    if (j < n) {
      const u32 i = d.perm[j];
      const u32 o0 = d.off[i];
      len = d.off[i + 1] - o0;
      src = d.pay + o0;
      dst = d.out_pay + d.ppos[j];
      if (d.ppos[j] + len > d.max_pay) len = 0;
    }
    int32_t v[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const u32 k = sub + 8 * q;
      v[q] = (k < len) ? src[k] : 0;
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const u32 k = sub + 8 * q;
      if (k < len) dst[k] = v[q];
    }
    for (u32 k = 64 + sub; k < len; k += 8) dst[k] = src[k];
  }
}

__global__ void k_rt_end(Ctl* ctl) {
  pdl_enter();
  if (ctl->status != ALTO_OK) return;
  if (ctl->batch_err) ctl->status = -(ctl->batch_err & 0xFF);
}

// Forget the flows of completed groups at the routing level: the slot
// becomes a tombstone (its replica and first fragment back to kNone), then
// runs of tombstones that end at a free slot become free (no probe chain
// runs through them).
__global__ void __launch_bounds__(kRT) k_rt_release(RDev d, const alto_record* rec, u64 n_rec) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (halted(ctl)) return;
  for (u64 k = blockIdx.x * (u64)blockDim.x + threadIdx.x; k < n_rec; k += gridDim.x * (u64)blockDim.x) {
    if ((int)rec[k].level != d.level) continue;
    const u64 key = ((u64)d.level << 32) | rec[k].parent_id;
    u32 h = (u32)mix64(key) & d.fmask;
    for (int p = 0; p < d.fprobe; ++p) {
      const u64 cur = d.fkey[h];
      if (cur == kEmpty) break;
      if (cur == key) {
        d.frep[h] = kNone;
        d.ffirst[h] = kNone;
        d.fkey[h] = kTomb;
        const u32 pos = atomicAdd(&ctl->n_done, 1u);
        if (pos < d.nmax) d.freed[pos] = h;
        break;
      }
      h = (h + 1) & d.fmask;
    }
  }
}

__global__ void __launch_bounds__(kRT) k_rt_sweep(RDev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  const u32 nf = min(ctl->n_done, d.nmax);
  volatile u64* key = d.fkey;
  for (u32 k = blockIdx.x * blockDim.x + threadIdx.x; k < nf; k += gridDim.x * blockDim.x) {
    const u32 e = d.freed[k];
    if (key[e] != kTomb) continue;
    u32 p = (e + 1) & d.fmask;
    int steps = 0;
    while (key[p] == kTomb && steps < d.fprobe) {
      p = (p + 1) & d.fmask;
      ++steps;
    }
    if (key[p] != kEmpty) continue;
    key[e] = kEmpty;
    u32 q = (e - 1) & d.fmask;
    steps = 0;
    while (key[q] == kTomb && steps < d.fprobe) {
      key[q] = kEmpty;
      q = (q - 1) & d.fmask;
      ++steps;
    }
  }
}

__global__ void k_rt_release_begin(Ctl* ctl) {
  pdl_enter();
  ctl->n_done = 0;
}

u64 next_pow2_rt(u64 x) {
  u64 p = 1;
  while (p < x) p <<= 1;
  return p;
}

int ilog2_rt(u64 x) {
  int b = 0;
  while ((1ull << b) < x) ++b;
  return b;
}

}  // namespace
}  // namespace alto

using namespace alto;

struct alto_router {
  alto_router_config cfg;
  alto_allocator alloc;
  bool use_async;
  int num_sms;
  RDev d;
  SortBuffers sb;
  LookbackState lbs;
  Ctl* h_ctl;
  std::vector<void*> blocks;
  int latched;
  int sort_bits;
};

namespace {

void* rt_alloc(alto_router* h, size_t bytes, cudaStream_t s) {
  bytes = std::max<size_t>((bytes + 255) & ~(size_t)255, 256);
  void* p = nullptr;
  if (h->use_async) {
    if (cudaMallocAsync(&p, bytes, s) != cudaSuccess) return nullptr;
  } else {
    p = h->alloc.alloc(h->alloc.ctx, bytes, s);
  }
  if (p) h->blocks.push_back(p);
  return p;
}

void rt_free_all(alto_router* h, cudaStream_t s) {
  for (void* p : h->blocks) {
    if (h->use_async) cudaFreeAsync(p, s);
    else h->alloc.free(h->alloc.ctx, p, s);
  }
  h->blocks.clear();
  if (h->h_ctl) cudaFreeHost(h->h_ctl);
  h->h_ctl = nullptr;
}

}  // namespace

extern "C" alto_status alto_router_create(const alto_router_config* cfg_in, const alto_allocator* alloc,
                                          void* stream, alto_router_t** out) {
  if (cfg_in == nullptr || out == nullptr) return ALTO_EINVAL;
  alto_router_config cfg = *cfg_in;
  if (cfg.depth < 1 || cfg.depth > ALTO_MAX_DEPTH || cfg.level < 0 || cfg.level >= cfg.depth) return ALTO_EINVAL;
  if (cfg.n_replicas < 1 || cfg.n_replicas > ALTO_MAX_REPLICAS) return ALTO_EINVAL;
  if (cfg.policy != ALTO_ROUTE_HASH && cfg.policy != ALTO_ROUTE_LEAST_LOADED) return ALTO_EINVAL;
  if (cfg.max_batch_fragments < 1 || cfg.max_batch_fragments >= (1ll << 30)) return ALTO_EINVAL;
  if (cfg.max_batch_payload < 0 || cfg.max_batch_payload >= (1ll << 32)) return ALTO_EINVAL;
  if (cfg.max_flows < 0 || cfg.max_flows > (1ll << 25)) return ALTO_EINVAL;
  if (alloc != nullptr && (alloc->alloc == nullptr || alloc->free == nullptr)) return ALTO_EINVAL;
  if (cfg.max_flows == 0) cfg.max_flows = 1ll << 20;
  cudaStream_t s = (cudaStream_t)stream;
  alto_router* h = new (std::nothrow) alto_router();
  if (!h) return ALTO_ENOMEM;
  h->cfg = cfg;
  h->use_async = (alloc == nullptr);
  if (alloc) h->alloc = *alloc;
  h->latched = ALTO_OK;
  h->h_ctl = nullptr;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      sort_prepare() != cudaSuccess) {
    delete h;
    return ALTO_ECUDA;
  }
  const u64 nmax = (u64)cfg.max_batch_fragments, R = (u64)cfg.n_replicas;
  const u64 T = next_pow2_rt(std::max<u64>(2 * (u64)cfg.max_flows, 1024));
  RDev& d = h->d;
  memset(&d, 0, sizeof(d));
  d.depth = cfg.depth;
  d.level = cfg.level;
  d.R = cfg.n_replicas;
  d.policy = cfg.policy;
  d.with_score = cfg.with_score ? 1 : 0;
  d.nmax = (u32)nmax;
  d.max_pay = (u64)cfg.max_batch_payload;
  d.fmask = (u32)(T - 1);
  d.fprobe = (int)std::min<u64>(T, 1u << 16);
  bool ok = true;
#define RALLOC(ptr, type, count)                                      \
  do {                                                                \
    ptr = (type*)rt_alloc(h, sizeof(type) * (size_t)(count), s);      \
    if (!ptr) ok = false;                                             \
  } while (0)
  RALLOC(d.ctl, Ctl, 1);
  if (cfg.policy == ALTO_ROUTE_LEAST_LOADED) {
    RALLOC(d.fkey, u64, T);
    RALLOC(d.frep, u32, T);
    RALLOC(d.ffirst, u32, T);
    RALLOC(d.freed, u32, nmax);
    RALLOC(d.fe, u32, nmax);
    RALLOC(d.rank, u32, nmax);
  }
  RALLOC(d.order, u32, R);
  RALLOC(d.load, u64, R);
  RALLOC(d.counts, u32, R);
  for (int b = 0; b < 2; ++b) {
    RALLOC(h->sb.keys[b], u32, nmax);
    RALLOC(h->sb.vals[b], u32, nmax);
  }
  const u64 sort_tiles = nmax / 4096 + 2;
  RALLOC(h->sb.hist, u32, 4 * 256);
  RALLOC(h->sb.bin_base, u32, 4 * 256);
  RALLOC(h->sb.lookback, u64, sort_tiles * 256);
  h->sb.lb_tiles = sort_tiles;
  d.rep_key = h->sb.keys[0];
  RALLOC(d.replica, u32, nmax);
  RALLOC(d.frag_off, int64_t, R + 1);
  RALLOC(d.pay_off, int64_t, R + 1);
  RALLOC(d.ppos, u64, nmax + 1);
  RALLOC(d.out_tags, u64, (u64)cfg.depth * nmax);
  RALLOC(d.out_poff, u32, nmax + R);
  RALLOC(d.out_pay, int32_t, std::max<u64>((u64)cfg.max_batch_payload, 1));
  if (cfg.with_score) RALLOC(d.out_score, float, nmax);
  const u64 scan_tiles = nmax / kScanTile + 2;
  RALLOC(h->lbs.desc, ulonglong2, scan_tiles);
  h->lbs.tiles = scan_tiles;
#undef RALLOC
  if (ok && cudaMallocHost((void**)&h->h_ctl, sizeof(Ctl)) != cudaSuccess) {
    h->h_ctl = nullptr;
    ok = false;
  }
  if (!ok) {
    rt_free_all(h, s);
    cudaStreamSynchronize(s);
    delete h;
    return ALTO_ENOMEM;
  }
  h->sort_bits = std::max(ilog2_rt(R), 1);
  cudaMemsetAsync(d.ctl, 0, sizeof(Ctl), s);
  if (d.fkey) {
    cudaMemsetAsync(d.fkey, 0xFF, sizeof(u64) * T, s);
    cudaMemsetAsync(d.frep, 0xFF, sizeof(u32) * T, s);
    cudaMemsetAsync(d.ffirst, 0xFF, sizeof(u32) * T, s);
  }
  cudaMemsetAsync(d.load, 0, sizeof(u64) * R, s);
  cudaMemsetAsync(h->sb.hist, 0, sizeof(u32) * 4 * 256, s);
  cudaMemsetAsync(h->sb.lookback, 0, sizeof(u64) * sort_tiles * 256, s);
  cudaMemsetAsync(h->lbs.desc, 0, sizeof(ulonglong2) * scan_tiles, s);
  if (cudaGetLastError() != cudaSuccess) {
    rt_free_all(h, s);
    delete h;
    return ALTO_ECUDA;
  }
  *out = h;
  return ALTO_OK;
}

extern "C" alto_status alto_router_route(alto_router_t* h, const alto_batch* b, void* stream, alto_routed* out) {
  if (h == nullptr || b == nullptr || out == nullptr) return ALTO_EINVAL;
  if (h->latched != ALTO_OK) return h->latched;
  const alto_router_config& cfg = h->cfg;
  if (b->depth != cfg.depth || b->n < 0 || b->n > cfg.max_batch_fragments) return ALTO_EINVAL;
  if (b->n_payload < 0 || b->n_payload > cfg.max_batch_payload) return ALTO_EINVAL;
  if (b->n > 0 && (b->tags == nullptr || b->payload_off == nullptr)) return ALTO_EINVAL;
  if (b->n_payload > 0 && b->payload == nullptr) return ALTO_EINVAL;
  if (b->n > 0 && cfg.with_score && b->score == nullptr) return ALTO_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  RDev d = h->d;
  d.tags = b->tags;
  d.off = b->payload_off;
  d.pay = b->payload;
  d.score = b->score;
  d.n = (u32)b->n;
  d.n_payload = (u64)b->n_payload;
  const int grid = h->num_sms * 8;
  const u64 spin = 1ull << 20;
  launch_pdl(k_rt_begin, 1, 1024, 0, s, d, (u32)b->n);
  launch_pdl(k_rt_assign, grid, kRT, 0, s, d);
  if (cfg.policy == ALTO_ROUTE_LEAST_LOADED) {
    RankScan2 f{d};
    const u64 tiles = std::max<u64>(((u64)cfg.max_batch_fragments + kScanTile - 1) / kScanTile, 1);
    launch_pdl(k_scan<RankScan2>, (int)std::min<u64>(tiles, (u64)h->num_sms * 4), kScanThreads, 0, s, f,
               h->lbs, d.ctl, 8, &d.ctl->exit_ctr[8], spin);
    launch_pdl(k_rt_order, 1, 1024, 0, s, d);
    launch_pdl(k_rt_place, grid, kRT, 0, s, d);
  }
  launch_pdl(k_rt_final, grid, kRT, 0, s, d);
  launch_pdl(k_rt_offsets, 1, 1024, 0, s, d);
  // stable partition by replica
  if (cfg.n_replicas > 1) {
    int sl = 0;
    const int cur = sort_pairs(&d.ctl->n, (u32)cfg.max_batch_fragments, h->sort_bits, true, h->sb, d.ctl, 0,
                               spin, h->num_sms, s, &sl);
    d.perm = h->sb.vals[cur];
    d.skey = h->sb.keys[cur];
  } else {
    launch_pdl(k_rt_identity, grid, kRT, 0, s, d, h->sb.vals[0]);
    d.perm = h->sb.vals[0];
    d.skey = nullptr;
  }
  {
    PermLenScan f{d};
    const u64 tiles = std::max<u64>(((u64)cfg.max_batch_fragments + kScanTile - 1) / kScanTile, 1);
    launch_pdl(k_scan<PermLenScan>, (int)std::min<u64>(tiles, (u64)h->num_sms * 4), kScanThreads, 0, s, f,
               h->lbs, d.ctl, 9, &d.ctl->exit_ctr[9], spin);
  }
  launch_pdl(k_rt_scatter, grid, kRT, 0, s, d);
  launch_pdl(k_rt_copy, grid, kRT, 0, s, d);
  launch_pdl(k_rt_end, 1, 1, 0, s, d.ctl);
  if (cudaGetLastError() != cudaSuccess) return ALTO_ECUDA;
  out->replica = d.replica;
  out->perm = d.perm;
  out->frag_off = d.frag_off;
  out->pay_off = d.pay_off;
  out->tags = d.out_tags;
  out->payload_off = d.out_poff;
  out->payload = d.out_pay;
  out->score = cfg.with_score ? d.out_score : nullptr;
  return ALTO_OK;
}

extern "C" alto_status alto_router_counts(alto_router_t* h, void* stream, int64_t* frag_off, int64_t* pay_off) {
  if (h == nullptr) return ALTO_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  const size_t nb = sizeof(int64_t) * (size_t)(h->cfg.n_replicas + 1);
  if (cudaMemcpyAsync(h->h_ctl, h->d.ctl, sizeof(Ctl), cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return ALTO_ECUDA;
  if (frag_off && cudaMemcpyAsync(frag_off, h->d.frag_off, nb, cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return ALTO_ECUDA;
  if (pay_off && cudaMemcpyAsync(pay_off, h->d.pay_off, nb, cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return ALTO_ECUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return ALTO_ECUDA;
  if (h->h_ctl->status != ALTO_OK) h->latched = h->h_ctl->status;
  return h->h_ctl->status;
}

extern "C" alto_status alto_router_release(alto_router_t* h, const alto_record* records, int64_t n_records,
                                           void* stream) {
  if (h == nullptr || n_records < 0 || (n_records > 0 && records == nullptr)) return ALTO_EINVAL;
  if (h->latched != ALTO_OK) return h->latched;
  if (h->cfg.policy != ALTO_ROUTE_LEAST_LOADED || n_records == 0) return ALTO_OK;
  cudaStream_t s = (cudaStream_t)stream;
  const int grid = h->num_sms * 2;
  launch_pdl(k_rt_release_begin, 1, 1, 0, s, h->d.ctl);
  launch_pdl(k_rt_release, grid, kRT, 0, s, h->d, records, (u64)n_records);
  launch_pdl(k_rt_sweep, grid, kRT, 0, s, h->d);
  if (cudaGetLastError() != cudaSuccess) return ALTO_ECUDA;
  return ALTO_OK;
}

extern "C" alto_status alto_router_destroy(alto_router_t* h) {
  if (h == nullptr) return ALTO_OK;
  cudaDeviceSynchronize();
  rt_free_all(h, nullptr);
  cudaDeviceSynchronize();
  delete h;
  return ALTO_OK;
}
