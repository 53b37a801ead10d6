// split_text: the fragmentation step in front of the aggregator (Alto, arxiv
// 2403.04311, Sec. 3.1-3.2: split_text turns a text item of a Delimiter type
// into a stream of smaller Delimiter items; Sec. 4.2: at a pmap entry every
// child keeps its parent's tags and gets one new tag), on one GB300.
//
// After the scratch is cleared, three launches:
//   mark    per stream: check its offsets, flag its last token
//   count   piece ends over the tokens (a delimiter, or a stream's last
//           token): a reduce-then-scan, two streaming passes (a look-back scan
//           would walk back a whole wave of tiles at 100M tokens); empty
//           streams over the streams: a look-back scan
//   write   per piece end, and per empty stream: the piece's fragment index
//           (piece ends before it + empty streams before its stream), its
//           tags, and its end offset.  Pieces tile the token buffer, so a
//           piece starts where the previous one ends and nothing is copied.
#include <cuda_runtime.h>

#include <algorithm>

#include "alto_agg.h"
#include "common.cuh"
#include "kernels.h"
#include "scan.cuh"

namespace alto {
namespace {

constexpr int kSplitThreads = 256;

struct SplitDev {
  Ctl* ctl;
  int32_t delims[ALTO_MAX_DELIMS];
  int n_delims;
  int depth_in;
  u64 n_src, n_tokens, cap;
  const u64* src_tags;
  const u32* src_id;
  const u32* tok_off;
  const int32_t* tokens;
  unsigned char* endmark;  // [n_tokens] last token of a non-empty stream
  u32* ends;    // [n_tokens + 1] piece ends before each token
  u32* empt;    // [n_src + 1] empty streams before each stream
  u64* out_tags;
  u32* out_off;
  int64_t* out_counts;
};

// A loop over the delimiters actually given (one to a few): every token
// passes through here twice, so a fully unrolled check of all 32 slots would
// make both passes instruction-bound.
__device__ __forceinline__ bool is_delim(const SplitDev& d, int32_t t) {
  for (int k = 0; k < d.n_delims; ++k)
    if (t == d.delims[k]) return true;
  return false;
}

__global__ void k_split_begin(Ctl* ctl) {
  pdl_enter();
  ctl->epoch = 1;
  ctl->status = ALTO_OK;
  ctl->batch_err = 0;
  ctl->abort = 0;
}

// Per stream: offsets must start at 0, not decrease and end at n_tokens.
__global__ void __launch_bounds__(kSplitThreads) k_split_mark(SplitDev d) {
  pdl_enter();
  for (u64 s = (u64)blockIdx.x * blockDim.x + threadIdx.x; s < d.n_src; s += (u64)gridDim.x * blockDim.x) {
    const u32 a = d.tok_off[s], b = d.tok_off[s + 1];
    bool bad = b < a || b > d.n_tokens;
    if (s == 0 && a != 0) bad = true;
    if (s + 1 == d.n_src && b != d.n_tokens) bad = true;
    if (bad) {
      raise_err(d.ctl, ALTO_EINVAL);
      continue;
    }
    if (b > a) d.endmark[b - 1] = 1;
  }
}

// which 0: piece ends over the tokens; 1: empty streams over the streams; 2: none
struct SplitScan {
  SplitDev d;
  int which;
  __device__ u64 size(const Ctl*) const { return (which == 0) ? d.n_tokens : (which == 1) ? d.n_src : 0; }
  __device__ u64 value(u64 i) const {
    if (which == 0) return (is_delim(d, d.tokens[i]) || d.endmark[i]) ? 1u : 0u;
    return (d.tok_off[i + 1] == d.tok_off[i]) ? 1u : 0u;
  }
  __device__ void out(u64 i, u64 excl, u64) const {
    if (which == 0) d.ends[i] = (u32)excl;
    else if (which == 1) d.empt[i] = (u32)excl;
  }
  __device__ void total(Ctl* ctl, u64 t) const {
    if (which == 0) d.ends[d.n_tokens] = (u32)t;
    else if (which == 1) d.empt[d.n_src] = (u32)t;
    if (which < 2) ctl->scan_total[which] = t;
  }
};

// Piece f (of `stride`) of stream s, ending at token `end`; `first` is the
// stream's first piece index.
__device__ __forceinline__ void put_piece(const SplitDev& d, u64 stride, u64 s, u64 f, u32 end, bool last,
                                          u64 first) {
  d.out_off[f + 1] = end;
  for (int l = 0; l < d.depth_in; ++l) d.out_tags[(u64)l * stride + f] = d.src_tags[(u64)l * d.n_src + s];
  d.out_tags[(u64)d.depth_in * stride + f] =
      ((u64)d.src_id[s] << 32) | ((u64)(last ? 1u : 0u) << 31) | ((f - first) & 0x7FFFFFFFull);
}

// Each warp takes one contiguous range of tokens: lane 0 finds the stream of
// its first token by binary search once, and the warp steps forward from
// there, 32 tokens at a time (four rounds' loads in flight).  A piece's index
// is the range's first index (one load) plus the pieces the warp has ended
// since (ballots), and the current stream's first piece index is kept in
// registers, so a piece costs no dependent load of its own; the next step's
// tokens are loaded before this step's pieces are written.
constexpr int kSplitRounds = 4;

__global__ void __launch_bounds__(kSplitThreads) k_split_write(SplitDev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  const u64 n_frag = ctl->scan_total[0] + ctl->scan_total[1];
  const bool ok = ctl->batch_err == 0 && *(volatile int*)&ctl->abort == 0;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    d.out_counts[0] = !ok ? -(ctl->batch_err & 0xFF) : (n_frag > d.cap ? ALTO_ENOSPC : ALTO_OK);
    if (!ok && ctl->batch_err == 0) d.out_counts[0] = ALTO_ETIMEOUT;
    d.out_counts[1] = (int64_t)n_frag;
    if (ok && n_frag <= d.cap) d.out_off[0] = 0;
  }
  if (!ok || n_frag > d.cap) return;
  const int lane = threadIdx.x & 31;
  const u64 gw = ((u64)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const u64 nw = ((u64)gridDim.x * blockDim.x) >> 5;
  const u64 step = 32ull * kSplitRounds;
  const u64 per = (d.n_tokens + nw - 1) / nw;
  const u64 lo = min(d.n_tokens, (per + step - 1) / step * step * gw);
  const u64 hi = min(d.n_tokens, lo + (per + step - 1) / step * step);
  u64 s = 0;
  if (lo < hi) {
    if (lane == 0) {
      u64 a = 0, b = d.n_src;  // last stream with tok_off[s] <= lo
      while (b - a > 1) {
        const u64 mid = (a + b) >> 1;
        if (d.tok_off[mid] <= lo) a = mid;
        else b = mid;
      }
      s = a;
    }
    s = __shfl_sync(0xFFFFFFFFu, s, 0);
  }
  // pieces ended before this warp's range, and the current stream's first piece
  u64 done = (lo < hi) ? (u64)d.ends[lo] : 0;
  u64 first_s = (lo < hi) ? (u64)d.ends[d.tok_off[s]] + d.empt[s] : 0;
  u32 empt_s = (lo < hi) ? d.empt[s] : 0;
  bool end[kSplitRounds];
#pragma unroll
  for (int r = 0; r < kSplitRounds; ++r) {
    const u64 p = lo + 32ull * r + lane;
    end[r] = p < hi && (is_delim(d, d.tokens[p]) || d.endmark[p]);
  }
  for (u64 base = lo; base < hi; base += step) {
    u32 m[kSplitRounds];
#pragma unroll
    for (int r = 0; r < kSplitRounds; ++r) m[r] = __ballot_sync(0xFFFFFFFFu, end[r]);
    // the next step's tokens go out before this step's pieces are written
    const u64 nb = base + step;
#pragma unroll
    for (int r = 0; r < kSplitRounds; ++r) {
      const u64 p = nb + 32ull * r + lane;
      end[r] = p < hi && (is_delim(d, d.tokens[p]) || d.endmark[p]);
    }
#pragma unroll
    for (int r = 0; r < kSplitRounds; ++r) {
      const u64 p = base + 32ull * r + lane;
      if ((m[r] >> lane) & 1u) {
        u64 sp = s;
        while (sp + 1 < d.n_src && d.tok_off[sp + 1] <= p) ++sp;
        const u64 k = done + __popc(m[r] & lanemask_lt());  // = ends[p]
        const u32 em = (sp == s) ? empt_s : d.empt[sp];
        const u64 fs = (sp == s) ? first_s : (u64)d.ends[d.tok_off[sp]] + d.empt[sp];
        put_piece(d, n_frag, sp, k + em, (u32)(p + 1), p + 1 == d.tok_off[sp + 1], fs);
      }
      done += __popc(m[r]);
    }
    // the stream of the next step's first token
    const u64 s0 = s;
    while (s + 1 < d.n_src && d.tok_off[s + 1] <= nb) ++s;
    if (s != s0 && nb < hi) {
      empt_s = d.empt[s];
      first_s = (u64)d.ends[d.tok_off[s]] + empt_s;
    }
  }
  for (u64 st = (u64)blockIdx.x * blockDim.x + threadIdx.x; st < d.n_src; st += (u64)gridDim.x * blockDim.x) {
    const u32 a = d.tok_off[st];
    if (d.tok_off[st + 1] != a) continue;
    const u64 f = (u64)d.ends[a] + d.empt[st];
    put_piece(d, n_frag, st, f, a, true, f);
  }
}

u64 align256(u64 x) { return (x + 255) & ~255ull; }

struct SplitLayout {
  u64 ctl, desc, ends, empt, mark, total;
  u64 tiles;
};

SplitLayout split_layout(u64 n_src, u64 n_tokens) {
  SplitLayout L;
  L.tiles = std::max(n_src, n_tokens) / kScanTile + 2;
  u64 o = 0;
  L.ctl = o;
  o += align256(sizeof(Ctl));
  L.desc = o;
  o += align256(3 * L.tiles * sizeof(ulonglong2));
  L.ends = o;
  o += align256((n_tokens + 1) * sizeof(u32));
  L.empt = o;
  o += align256((n_src + 1) * sizeof(u32));
  L.mark = o;
  o += align256(std::max<u64>(n_tokens, 1));
  L.total = o;
  return L;
}

}  // namespace
}  // namespace alto

using namespace alto;

extern "C" int64_t alto_split_scratch_bytes(int64_t n_src, int64_t n_tokens) {
  if (n_src < 1 || n_tokens < 0) return 0;
  return (int64_t)split_layout((u64)n_src, (u64)n_tokens).total;
}

extern "C" alto_status alto_split_text(const alto_split_args* a, void* stream) {
  if (a == nullptr) return ALTO_EINVAL;
  if (a->n_src < 1 || a->n_tokens < 0 || a->n_tokens >= (1ll << 32) || a->n_src >= (1ll << 32))
    return ALTO_EINVAL;
  if (a->depth_in < 0 || a->depth_in >= ALTO_MAX_DEPTH) return ALTO_EINVAL;
  if (a->n_delims < 1 || a->n_delims > ALTO_MAX_DELIMS || a->cap_frag < 0) return ALTO_EINVAL;
  if (a->src_id == nullptr || a->tok_off == nullptr || a->out_off == nullptr || a->out_tags == nullptr ||
      a->out_counts == nullptr || a->scratch == nullptr || (a->n_tokens > 0 && a->tokens == nullptr) ||
      (a->depth_in > 0 && a->src_tags == nullptr))
    return ALTO_EINVAL;
  if ((((uintptr_t)a->scratch) & 255) != 0) return ALTO_EINVAL;
  const SplitLayout L = split_layout((u64)a->n_src, (u64)a->n_tokens);
  if (a->scratch_bytes < (int64_t)L.total) return ALTO_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  unsigned char* base = (unsigned char*)a->scratch;
  SplitDev d;
  d.ctl = (Ctl*)(base + L.ctl);
  for (int k = 0; k < ALTO_MAX_DELIMS; ++k) d.delims[k] = (k < a->n_delims) ? a->delims[k] : 0;
  d.n_delims = a->n_delims;
  d.depth_in = a->depth_in;
  d.n_src = (u64)a->n_src;
  d.n_tokens = (u64)a->n_tokens;
  d.cap = (u64)a->cap_frag;
  d.src_tags = a->src_tags;
  d.src_id = a->src_id;
  d.tok_off = a->tok_off;
  d.tokens = a->tokens;
  d.endmark = base + L.mark;
  d.ends = (u32*)(base + L.ends);
  d.empt = (u32*)(base + L.empt);
  d.out_tags = a->out_tags;
  d.out_off = a->out_off;
  d.out_counts = a->out_counts;
  LookbackState lb;
  lb.desc = (ulonglong2*)(base + L.desc);
  lb.tiles = L.tiles;
  // the control block, the look-back descriptors and the last-token marks start empty
  cudaMemsetAsync(base + L.ctl, 0, L.ends - L.ctl, s);
  cudaMemsetAsync(base + L.mark, 0, std::max<u64>(d.n_tokens, 1), s);
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return ALTO_ECUDA;
  const u64 spin = 1ull << 20;
  launch_pdl(k_split_begin, 1, 1, 0, s, d.ctl);
  const int sgrid = (int)std::min<u64>((d.n_src + kSplitThreads - 1) / kSplitThreads + 1, (u64)sms * 8);
  launch_pdl(k_split_mark, sgrid, kSplitThreads, 0, s, d);
  {
    // streams: a look-back scan over the first descriptor region; tokens: a
    // reduce-then-scan whose chunk sums live in the second region
    SplitScan fs{d, 1}, ft{d, 0};
    const u64 stiles = std::max<u64>((d.n_src + kScanTile - 1) / kScanTile, 1);
    launch_pdl(k_scan<SplitScan>, (int)std::min<u64>(stiles, (u64)sms * 4), kScanThreads, 0, s, fs, lb,
               d.ctl, 1, &d.ctl->exit_ctr[1], spin);
    u64* part = reinterpret_cast<u64*>(lb.desc + lb.tiles);
    const int rgrid = (int)std::min<u64>((u64)sms * 4, 2 * lb.tiles);
    launch_pdl(k_scan_reduce<SplitScan>, rgrid, kScanThreads, 0, s, ft, part, d.ctl);
    launch_pdl(k_scan_down<SplitScan>, rgrid, kScanThreads, 0, s, ft, (const u64*)part, d.ctl);
  }
  // every warp owns a fixed token range: the grid is exactly the warps that
  // fit on the GPU at once (a second wave would run its ranges after the first)
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_split_write, kSplitThreads, 0) != cudaSuccess ||
      per_sm < 1)
    per_sm = 1;
  launch_pdl(k_split_write, sms * per_sm, kSplitThreads, 0, s, d);
  if (cudaGetLastError() != cudaSuccess) return ALTO_ECUDA;
  return ALTO_OK;
}
