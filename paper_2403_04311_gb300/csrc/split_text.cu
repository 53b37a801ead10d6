// split_text: the fragmentation step in front of the aggregator (Alto, arxiv
// 2403.04311, Sec. 3.1-3.2: split_text turns a text item of a Delimiter type
// into a stream of smaller Delimiter items; Sec. 4.2: at a pmap entry every
// child keeps its parent's tags and gets one new tag), on one GB300.
//
// After the scratch is cleared:
//   mark    per stream: check its offsets, flag its last token
//   empty   empty streams before each stream (a look-back scan over streams)
//   count   every warp owns one contiguous range of tokens and counts the
//           piece ends in it (a delimiter, or a stream's last token), and for
//           every stream starting in it the ends before that start
//   ranges  the ends before each range (a look-back scan over the ranges)
//   write   per piece end, and per empty stream: the piece's fragment index
//           (piece ends before it + empty streams before its stream), its
//           tags, and its end offset.  Pieces tile the token buffer, so a
//           piece starts where the previous one ends and nothing is copied.
// The tokens are read twice (count, write); no per-token array is written.
#include <cuda_runtime.h>

#include <algorithm>

#include "alto_agg.h"
#include "common.cuh"
#include "kernels.h"
#include "scan.cuh"

namespace alto {
namespace {

constexpr int kSplitThreads = 256;

// count and write split the tokens into the same ranges, one a warp
constexpr int kSplitRounds = 4;         // rounds of loads a warp keeps in flight
constexpr u64 kSplitRound = 128;        // tokens a round: four consecutive ones a lane
constexpr u64 kSplitStep = kSplitRounds * kSplitRound;
constexpr u64 kSplitMaxWarps = 1u << 15;

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
  u32* empt;    // [n_src + 1] empty streams before each stream
  u32* sloc;    // [n_src] piece ends between its range's first token and the stream's first token
  u32* wcnt;    // [nwarps] piece ends in each range
  u32* wpre;    // [nwarps + 1] piece ends before each range
  u64 range;    // tokens per range (a multiple of kSplitStep)
  u32 nwarps;
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

// which 0: piece ends before each range; 1: empty streams over the streams
struct SplitScan {
  SplitDev d;
  int which;
  __device__ u64 size(const Ctl*) const { return (which == 0) ? d.nwarps : d.n_src; }
  __device__ u64 value(u64 i) const {
    if (which == 0) return d.wcnt[i];
    return (d.tok_off[i + 1] == d.tok_off[i]) ? 1u : 0u;
  }
  __device__ void out(u64 i, u64 excl, u64) const {
    if (which == 0) d.wpre[i] = (u32)excl;
    else d.empt[i] = (u32)excl;
  }
  __device__ void total(Ctl* ctl, u64 t) const {
    if (which == 0) d.wpre[d.nwarps] = (u32)t;
    else d.empt[d.n_src] = (u32)t;
    ctl->scan_total[which] = t;
  }
};

// The range [lo, hi) of warp w.
__device__ __forceinline__ void split_range(const SplitDev& d, u64 w, u64* lo, u64* hi) {
  *lo = min(d.n_tokens, w * d.range);
  *hi = min(d.n_tokens, *lo + d.range);
}

// Piece ends before token a, the first token of a stream s (a < n_tokens:
// its range's count before the range plus the stream's own count in it).
__device__ __forceinline__ u64 ends_before_start(const SplitDev& d, u64 s, u64 a) {
  return (a < d.n_tokens) ? (u64)d.wpre[a / d.range] + d.sloc[s] : (u64)d.wpre[d.nwarps];
}

// The end flags of the step at `base`: in round r, lane l owns tokens
// base + 128r + 4l .. +3 (bit k of f[r]: token 4l + k; none past hi).  With a
// 16-byte aligned token buffer a lane reads its four tokens and their four
// last-token marks with one load each.
__device__ __forceinline__ u32 end_bit(const SplitDev& d, int32_t tok, u32 mark) {
  return (is_delim(d, tok) || mark) ? 1u : 0u;
}
__device__ __forceinline__ void load_flags(const SplitDev& d, u64 base, u64 hi, bool vec, u32 (&f)[kSplitRounds]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int r = 0; r < kSplitRounds; ++r) {
    const u64 p = base + kSplitRound * r + 4ull * lane;
    u32 m = 0;
    if (vec && p + 4 <= hi) {
      const int4 t = *reinterpret_cast<const int4*>(d.tokens + p);
      const u32 mk = *reinterpret_cast<const u32*>(d.endmark + p);
      m = end_bit(d, t.x, mk & 0xFFu) | (end_bit(d, t.y, (mk >> 8) & 0xFFu) << 1) |
          (end_bit(d, t.z, (mk >> 16) & 0xFFu) << 2) | (end_bit(d, t.w, mk >> 24) << 3);
    } else {
      for (int k = 0; k < 4; ++k)
        if (p + k < hi) m |= end_bit(d, d.tokens[p + k], d.endmark[p + k]) << k;
    }
    f[r] = m;
  }
}

// Per round: the ends of the lanes before this one, and the round's total.
__device__ __forceinline__ void round_counts(const u32 (&f)[kSplitRounds], u32 (&excl)[kSplitRounds],
                                             u32 (&tot)[kSplitRounds]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int r = 0; r < kSplitRounds; ++r) {
    const u32 c = __popc(f[r]);
    u32 incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const u32 y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += y;
    }
    excl[r] = incl - c;
    tot[r] = __shfl_sync(0xFFFFFFFFu, incl, 31);
  }
}

// First stream whose first token is at or after `lo`.
__device__ __forceinline__ u64 first_stream_from(const SplitDev& d, u64 lo) {
  u64 a = 0, b = d.n_src;
  while (a < b) {
    const u64 mid = (a + b) >> 1;
    if (d.tok_off[mid] < lo) a = mid + 1;
    else b = mid;
  }
  return a;
}

// Per range: its piece ends, and for every stream starting in it the ends
// between the range's first token and the stream's first token.
__global__ void __launch_bounds__(kSplitThreads) k_split_count(SplitDev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (ctl->batch_err != 0 || *(volatile int*)&ctl->abort != 0) return;
  const int lane = threadIdx.x & 31;
  const u64 w = ((u64)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (w >= d.nwarps) return;
  u64 lo, hi;
  split_range(d, w, &lo, &hi);
  u64 ns = 0;  // next stream to start in this range
  if (lo < hi) {
    if (lane == 0) ns = first_stream_from(d, lo);
    ns = __shfl_sync(0xFFFFFFFFu, ns, 0);
  }
  const bool vec = (reinterpret_cast<uintptr_t>(d.tokens) & 15) == 0;
  u32 done = 0;
  u32 f[kSplitRounds];
  load_flags(d, lo, hi, vec, f);
  for (u64 base = lo; base < hi; base += kSplitStep) {
    u32 excl[kSplitRounds], tot[kSplitRounds], fc[kSplitRounds];
    round_counts(f, excl, tot);
#pragma unroll
    for (int r = 0; r < kSplitRounds; ++r) fc[r] = f[r];
    load_flags(d, base + kSplitStep, hi, vec, f);  // the next step's loads go out now
    const u64 top = min(base + kSplitStep, hi);
    while (ns < d.n_src && d.tok_off[ns] < top) {
      const u32 t = (u32)(d.tok_off[ns] - base);
      const u32 rr = t / (u32)kSplitRound, ll = (t % (u32)kSplitRound) >> 2, kk = t & 3u;
      u32 c = done;
#pragma unroll
      for (int r = 0; r < kSplitRounds; ++r) {
        const u32 ex = __shfl_sync(0xFFFFFFFFu, excl[r], ll);
        const u32 fl = __shfl_sync(0xFFFFFFFFu, fc[r], ll);
        if ((u32)r < rr) c += tot[r];
        else if ((u32)r == rr) c += ex + __popc(fl & ((1u << kk) - 1u));
      }
      if (lane == 0) d.sloc[ns] = c;
      ++ns;
    }
#pragma unroll
    for (int r = 0; r < kSplitRounds; ++r) done += tot[r];
  }
  if (lane == 0) d.wcnt[w] = done;
}

// Piece f (of `stride`) of stream s, ending at token `end`; `first` is the
// stream's first piece index.
__device__ __forceinline__ void put_piece(const SplitDev& d, u64 stride, u64 s, u64 f, u32 end, bool last,
                                          u64 first) {
  d.out_off[f + 1] = end;
  for (int l = 0; l < d.depth_in; ++l) d.out_tags[(u64)l * stride + f] = d.src_tags[(u64)l * d.n_src + s];
  d.out_tags[(u64)d.depth_in * stride + f] =
      ((u64)d.src_id[s] << 32) | ((u64)(last ? 1u : 0u) << 31) | ((f - first) & 0x7FFFFFFFull);
}

// Per range: each piece end's fragment index is the ends before the range
// (one load) plus the ends the warp has passed (ballots) plus the empty
// streams before its stream; the current stream's first piece index stays in
// registers, and the next step's tokens are loaded before this step's pieces
// are written.
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
  const u64 w = ((u64)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  u64 lo = 0, hi = 0;
  if (w < d.nwarps) split_range(d, w, &lo, &hi);
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
  u64 done = (lo < hi) ? (u64)d.wpre[w] : 0;
  u32 empt_s = (lo < hi) ? d.empt[s] : 0;
  u64 first_s = (lo < hi) ? ends_before_start(d, s, d.tok_off[s]) + empt_s : 0;
  const bool vec = (reinterpret_cast<uintptr_t>(d.tokens) & 15) == 0;
  u32 f[kSplitRounds];
  load_flags(d, lo, hi, vec, f);
  for (u64 base = lo; base < hi; base += kSplitStep) {
    u32 excl[kSplitRounds], tot[kSplitRounds], fc[kSplitRounds];
    round_counts(f, excl, tot);
#pragma unroll
    for (int r = 0; r < kSplitRounds; ++r) fc[r] = f[r];
    const u64 nb = base + kSplitStep;
    load_flags(d, nb, hi, vec, f);  // the next step's loads go out now
#pragma unroll
    for (int r = 0; r < kSplitRounds; ++r) {
      u32 bits = fc[r];
      u64 k = done + excl[r];  // piece ends before this lane's first token of the round
      while (bits) {
        const int b = __ffs(bits) - 1;
        bits &= bits - 1;
        const u64 p = base + kSplitRound * r + 4ull * lane + b;
        u64 sp = s;
        while (sp + 1 < d.n_src && d.tok_off[sp + 1] <= p) ++sp;
        const u32 em = (sp == s) ? empt_s : d.empt[sp];
        const u64 fs = (sp == s) ? first_s : ends_before_start(d, sp, d.tok_off[sp]) + em;
        put_piece(d, n_frag, sp, k + em, (u32)(p + 1), p + 1 == d.tok_off[sp + 1], fs);
        ++k;
      }
      done += tot[r];
    }
    // the stream of the next step's first token
    const u64 s0 = s;
    while (s + 1 < d.n_src && d.tok_off[s + 1] <= nb) ++s;
    if (s != s0 && nb < hi) {
      empt_s = d.empt[s];
      first_s = ends_before_start(d, s, d.tok_off[s]) + empt_s;
    }
  }
  for (u64 st = (u64)blockIdx.x * blockDim.x + threadIdx.x; st < d.n_src; st += (u64)gridDim.x * blockDim.x) {
    const u32 a = d.tok_off[st];
    if (d.tok_off[st + 1] != a) continue;
    const u64 f = ends_before_start(d, st, a) + d.empt[st];
    put_piece(d, n_frag, st, f, a, true, f);
  }
}

u64 align256(u64 x) { return (x + 255) & ~255ull; }

struct SplitLayout {
  u64 ctl, desc, empt, sloc, wcnt, wpre, mark, total;
  u64 tiles;
};

SplitLayout split_layout(u64 n_src, u64 n_tokens) {
  SplitLayout L;
  L.tiles = std::max<u64>(n_src, kSplitMaxWarps) / kScanTile + 2;
  u64 o = 0;
  L.ctl = o;
  o += align256(sizeof(Ctl));
  L.desc = o;
  o += align256(2 * L.tiles * sizeof(ulonglong2));
  L.empt = o;
  o += align256((n_src + 1) * sizeof(u32));
  L.sloc = o;
  o += align256(n_src * sizeof(u32));
  L.wcnt = o;
  o += align256(kSplitMaxWarps * sizeof(u32));
  L.wpre = o;
  o += align256((kSplitMaxWarps + 1) * sizeof(u32));
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
  d.empt = (u32*)(base + L.empt);
  d.sloc = (u32*)(base + L.sloc);
  d.wcnt = (u32*)(base + L.wcnt);
  d.wpre = (u32*)(base + L.wpre);
  d.out_tags = a->out_tags;
  d.out_off = a->out_off;
  d.out_counts = a->out_counts;
  LookbackState lb;
  lb.desc = (ulonglong2*)(base + L.desc);
  lb.tiles = L.tiles;
  // the control block and the look-back descriptors start empty, and so do
  // the last-token marks
  cudaMemsetAsync(base + L.ctl, 0, L.empt - L.ctl, s);
  cudaMemsetAsync(base + L.mark, 0, std::max<u64>(d.n_tokens, 1), s);
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return ALTO_ECUDA;
  // count and write give every warp one fixed token range: the grid is
  // exactly the warps that fit on the GPU at once (a second wave would run
  // its ranges after the first)
  int pc = 0, pw = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&pc, k_split_count, kSplitThreads, 0) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&pw, k_split_write, kSplitThreads, 0) != cudaSuccess)
    return ALTO_ECUDA;
  const u64 wpb = kSplitThreads / 32;
  const u64 blocks = std::max<u64>(1, std::min<u64>((u64)sms * (u64)std::max(1, std::min(pc, pw)),
                                                      kSplitMaxWarps / wpb));
  d.nwarps = (u32)(blocks * wpb);
  const u64 per = (d.n_tokens + d.nwarps - 1) / d.nwarps;
  d.range = std::max<u64>(kSplitStep, (per + kSplitStep - 1) / kSplitStep * kSplitStep);
  const u64 spin = 1ull << 20;
  launch_pdl(k_split_begin, 1, 1, 0, s, d.ctl);
  const int sgrid = (int)std::min<u64>((d.n_src + kSplitThreads - 1) / kSplitThreads + 1, (u64)sms * 8);
  launch_pdl(k_split_mark, sgrid, kSplitThreads, 0, s, d);
  SplitScan fs{d, 1}, fw{d, 0};
  LookbackState lb1 = lb;
  lb1.desc += lb.tiles;
  const u64 stiles = std::max<u64>((d.n_src + kScanTile - 1) / kScanTile, 1);
  launch_pdl(k_scan<SplitScan>, (int)std::min<u64>(stiles, (u64)sms), kScanThreads, 0, s, fs, lb1, d.ctl, 1,
             &d.ctl->exit_ctr[1], spin);
  launch_pdl(k_split_count, (int)blocks, kSplitThreads, 0, s, d);
  const u64 wtiles = std::max<u64>((d.nwarps + kScanTile - 1) / kScanTile, 1);
  launch_pdl(k_scan<SplitScan>, (int)std::min<u64>(wtiles, (u64)sms), kScanThreads, 0, s, fw, lb, d.ctl, 0,
             &d.ctl->exit_ctr[0], spin);
  launch_pdl(k_split_write, (int)blocks, kSplitThreads, 0, s, d);
  if (cudaGetLastError() != cudaSuccess) return ALTO_ECUDA;
  return ALTO_OK;
}
