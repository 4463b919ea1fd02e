// Decode-batch expert FFN (bf16, at most 64 tokens per call): HBM-streaming, one CTA per block of
// 16 weight rows, token products on the tensor cores with mma.sync m16n8k16.
//
// F(x) = W2 (silu(W1 x) * (W3 x)) for each expert segment (Section 3.1, SwiGLU experts). At
// decode the selected experts' weights are the only large operand, so the kernels are built to
// read every weight byte once, in whole lines, with many loads in flight:
//  * a CTA item is RB blocks of 16 consecutive rows of W1 and W3 (GEMM13), or of 32 rows of W2
//    (GEMM2, two MMA tiles sharing the activation fragments), of one segment; its 8 warps are
//    RB x KS (KS = 8 / RB contraction slices per row block, chosen so every warp walks at least 8
//    chunks), each walking its slice 64 elements at a time; in each load instruction the 4 lanes
//    of a quad read 64 contiguous bytes of one row; slice k holds chunks k, k + KS, k + 2 KS, ...,
//    so at each step the KS warps of a row block read KS adjacent chunks (KS x 128 contiguous
//    bytes of every row) rather than KS chunks far apart;
//  * the 16 x 64 weight slab is the A operand of four m16n8k16 MMAs (the contraction order inside
//    a 64-wide chunk is permuted identically for A and B, which leaves every dot product intact);
//    the B operand is 8 tokens of the segment, so one A fragment serves up to 32 tokens per pass
//    (segments of more tokens take a second pass, whose weight reads hit L2);
//  * the 8 partial sums are added in shared memory in a fixed order (deterministic); GEMM13 then
//    applies silu(gate) * up and stores h in bf16; GEMM2 stores fp32 outputs. At small batches
//    GEMM2 also splits the contraction across `ksplit` CTAs (partial planes of o, summed in the
//    combine kernel) so that few selected experts still give every SM work.
// Items are spread over a persistent grid: claimed from a counter by the fused kernel (both GEMMs
// in one launch, the path of every forward without LoRA adapters), with static striding by the
// separate GEMM13 and GEMM2 kernels (the LoRA forward, whose down projection of h sits between).
// Two CTAs of these kernels take all of an SM's registers, so when an expert fetch kernel may run
// at the same time the caller reserves its slots: a grid that took them would keep the fetch from
// starting until the FFN's CTAs exit.
#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

constexpr int kWarps = 8;
constexpr int kRows = 16;        // weight rows per warp (GEMM13: one MMA tile)
constexpr int kRows2 = 32;       // weight rows per warp (GEMM2: two MMA tiles)
constexpr int kChunk = 64;       // contraction elements per step (128 bytes of a row)
constexpr int kPassTokens = 32;  // tokens per pass (4 MMA column groups of 8)
constexpr int kMaxNG = kPassTokens / 8;

struct DecItems {
  int npos, total, ksplit, rb;  // rb: row blocks per item
  unsigned long long stream;    // segments streamed behind their fetch (seg_streamed)
  unsigned epoch;               // the stamp their landed pieces carry
  int off[kMaxSeg + 1];    // by segment: permuted-row offsets
  const char* blk[kMaxSeg];
  int seg[kMaxSeg];        // by position in the work list: segment
  int first[kMaxSeg + 1];  // by position: first item
};

// Work list of a launch, built by one warp (the calling one) with one lane per segment (segments
// s = lane, lane + 32, lane + 64): for every non-empty segment of the phase, its rows in items of
// rb blocks of rows_per_block rows, times ksplit contraction parts; segments in decreasing order
// of their token counts (ties by index), so that the items that take longest (segments that need
// a second pass or more MMA columns) are handed out first and the last ones are short; segments
// streamed behind their fetch come after all the others (their items wait for bytes still on the
// host link). Only segments with work get a position. The item shape depends on the layer and the batch only, not
// on which segments a launch computes, so an output is bit-identical whichever phase of a cached
// forward computes it. The caller synchronises the block before reading the list.
__device__ void build_dec_items(DecItems& it, const FfnArgs& a, int rows, int rows_per_block,
                                int rb, int ksplit, bool blk_ready = false) {
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  // every load first (abort flag, ready mask, offsets, block addresses: one round trip), then the
  // abort flag applied
  const int aborted = a.hdr->abort;
  const unsigned long long hits = a.ready ? *a.ready : 0ull;
  const unsigned long long stream = a.landed && a.stream ? *a.stream : 0ull;
  const unsigned epoch = a.landed ? static_cast<unsigned>(*a.epoch) : 0u;
  int offv[3];
  const char* blkv[3];
#pragma unroll
  for (int j = 0; j < 3; ++j) {
    const int s = lane + 32 * j;
    offv[j] = s <= a.nseg ? a.off[s] : 0;
    blkv[j] = s >= a.nseg ? nullptr
              : blk_ready ? it.blk[s] : reinterpret_cast<const char*>(seg_block(a, s));
  }
  const int nseg = aborted == 0 ? a.nseg : 0;
#pragma unroll
  for (int j = 0; j < 3; ++j) {
    const int s = lane + 32 * j;
    if (s <= nseg) it.off[s] = offv[j];
  }
  __syncwarp();
  bool bad = false;
  // key of a segment with work (else -1): its token count, raised by 2^20 unless it is streamed
  // behind its fetch, so that the streamed segments' items come last
  int key[3];
  unsigned work[3];
#pragma unroll
  for (int j = 0; j < 3; ++j) {
    const int s = lane + 32 * j;
    key[j] = -1;
    if (s < nseg) {
      const char* b = blkv[j];
      it.blk[s] = b;
      const int n = it.off[s + 1] - it.off[s];
      if (n > 0 && seg_in_phase(a, s, hits, stream)) {
        if (b == nullptr) bad = true;  // a selected expert without weights
        else key[j] = n + (seg_streamed(a, s, stream) ? 0 : (1 << 20));
      }
    }
    work[j] = __ballot_sync(full, key[j] >= 0);
  }
  const int npos = __popc(work[0]) + __popc(work[1]) + __popc(work[2]);
  const int items_per_seg = rows / (rows_per_block * rb);
  // position of each segment with work: those before it have more tokens, or as many and a lower
  // index (a strict total order, so the positions are 0 .. npos - 1, each taken once)
  int rank[3] = {0, 0, 0};
  for (int j2 = 0; j2 < 3; ++j2)
    for (unsigned m = work[j2]; m != 0u; m &= m - 1u) {
      const int src = __ffs(m) - 1, t = src + 32 * j2;
      const int kt = __shfl_sync(full, key[j2], src);
#pragma unroll
      for (int j = 0; j < 3; ++j)
        rank[j] += (kt > key[j] || (kt == key[j] && t < lane + 32 * j)) ? 1 : 0;
    }
  for (int j = 0; j < 3; ++j)
    if (key[j] >= 0) {
      it.seg[rank[j]] = lane + 32 * j;
      it.first[rank[j]] = items_per_seg * ksplit;  // the item count, until the scan below
    }
  __syncwarp();
  int base = 0;
  for (int j = 0; j < 3; ++j) {
    const int p = lane + 32 * j;
    const int c = p < npos ? it.first[p] : 0;
    int v = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int u = __shfl_up_sync(full, v, o);
      if (lane >= o) v += u;
    }
    if (p <= npos) it.first[p] = base + v - c;
    base += __shfl_sync(full, v, 31);
  }
  const bool any_bad = __any_sync(full, bad);
  if (lane == 0) {
    if (any_bad) {  // the other segments still run; later kernels of the call skip their work
      set_error(a.err, kErrInvalid);
      const_cast<WsHeader*>(a.hdr)->abort = 1;
    }
    it.npos = npos;
    it.ksplit = ksplit;
    it.rb = rb;
    it.total = base;
    it.stream = stream;
    it.epoch = epoch;
  }
}

// Threads t0 .. t0 + kMaxSeg - 1 of the block fill the segment block table of both work lists,
// one entry each. The fused kernel does this before its grid-dependency wait: the table comes from
// the kernel parameters and the cache's device table, written before the previous launch (the
// permutation, which lets this launch start early) began.
__device__ __forceinline__ void fill_blk(DecItems& x, DecItems& y, const FfnArgs& a, int t0) {
  const int s = int(threadIdx.x) - t0;
  if (s >= 0 && s < kMaxSeg) {
    const char* b = s < a.nseg ? reinterpret_cast<const char*>(seg_block(a, s)) : nullptr;
    x.blk[s] = b;
    y.blk[s] = b;
  }
}

// Position in the work list of an item (< it.total): the last position whose first item is at or
// before it.
__device__ __forceinline__ int dec_pos(const DecItems& it, int item) {
  int lo = 0, hi = it.npos - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (it.first[mid] <= item) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// A lane of quad position c holds elements 8c..8c+7 (lo) and 32+8c..32+8c+7 (hi) of a 64-wide
// chunk. MMA step j (0..3) uses 32-bit words 2j and 2j+1 of (lo, hi): for each c these are 4
// elements, and over the 4 lanes of the quad and the 4 steps every element is used exactly once.
__device__ __forceinline__ uint32_t word(const uint4& lo, const uint4& hi, int i) {
  switch (i) {
    case 0: return lo.x;
    case 1: return lo.y;
    case 2: return lo.z;
    case 3: return lo.w;
    case 4: return hi.x;
    case 5: return hi.y;
    case 6: return hi.z;
    default: return hi.w;
  }
}

// Walk chunks c0, c0 + step, ... below c1: load(buf, ch) issues a chunk's weight loads,
// compute(buf, ch) consumes them. With DB the next chunk's loads are issued before the current chunk's MMAs (two register
// buffers, unrolled by two so nothing is copied), so a warp keeps one chunk in flight while it
// computes; without DB each chunk is loaded, then consumed (token groups of more than 8, and any
// group in the kernel compiled for 32-token passes, whose accumulators need the registers).
template <bool DB, typename Load, typename Compute>
__device__ __forceinline__ void stream_chunks(int c0, int c1, int step, Load&& load,
                                              Compute&& compute) {
  uint4 va[8];
  if constexpr (DB) {
    uint4 vb[8];
    if (c0 < c1) load(va, c0);
    int ch = c0;
    for (; ch + step < c1; ch += 2 * step) {
      load(vb, ch + step);
      compute(va, ch);
      if (ch + 2 * step < c1) load(va, ch + 2 * step);
      compute(vb, ch + step);
    }
    if (ch < c1) compute(va, ch);
  } else {
    for (int ch = c0; ch < c1; ch += step) {
      load(va, ch);
      compute(va, ch);
    }
  }
}

// Chunks [c0, c1) of this warp's slice of a contraction of nch chunks.
__device__ __forceinline__ void warp_slice(int nch, int parts, int part, int& c0, int& c1) {
  const int per = (nch + parts - 1) / parts;
  c0 = min(nch, part * per);
  c1 = min(nch, c0 + per);
}

// GEMM13 + SwiGLU for RB blocks of 16 rows starting at r0 and n <= 32 tokens of one segment
// starting at permuted row q0; warp w owns row block w / KS and contraction slice w % KS
// (chunks w % KS, w % KS + KS, ...).
// red: shared scratch [kWarps][kMaxNG][8][32] floats.
// COH: weight loads through L2 only (ld.global.cg) for a block that a fetch kernel running beside
// this launch wrote; otherwise streaming non-coherent loads. Both read the same bytes.
template <bool COH>
__device__ __forceinline__ uint4 ldw16(const void* p) {
  if constexpr (COH) return ldcg16(p);
  else return ld_stream16(p);
}

template <int NG, bool DB, bool COH = false>
__device__ __forceinline__ void dec13_item(const FfnArgs& a, const char* blk, const void* lblk,
                                           int r0, int q0, int n, int RB, int KS, float* red) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const int rw = r0 + (warp / KS) * kRows;
  const size_t rowb = size_t(a.d) * 2;
  const char* w1g = blk + size_t(rw + g) * rowb + c * 16;
  const char* w1h = w1g + 8 * rowb;
  const char* w3g = blk + size_t(a.w + rw + g) * rowb + c * 16;
  const char* w3h = w3g + 8 * rowb;
  const char* xr[NG];
#pragma unroll
  for (int G = 0; G < NG; ++G) {
    const int j = G * 8 + g;
    const int t = a.perm[q0 + (j < n ? j : 0)];
    xr[G] = reinterpret_cast<const char*>(a.x) + size_t(t) * rowb + c * 16;
  }
  float accg[NG][4], accu[NG][4];
#pragma unroll
  for (int G = 0; G < NG; ++G)
#pragma unroll
    for (int i = 0; i < 4; ++i) accg[G][i] = accu[G][i] = 0.f;

  const int nch = int(rowb / (kChunk * 2));
  // one chunk's weights: W1 rows g / g+8 (lo, hi halves), then W3's
  auto load = [&](uint4* v, int ch) {
    const size_t k = size_t(ch) * kChunk * 2;
    v[0] = ldw16<COH>(w1g + k); v[1] = ldw16<COH>(w1g + k + 64);
    v[2] = ldw16<COH>(w1h + k); v[3] = ldw16<COH>(w1h + k + 64);
    v[4] = ldw16<COH>(w3g + k); v[5] = ldw16<COH>(w3g + k + 64);
    v[6] = ldw16<COH>(w3h + k); v[7] = ldw16<COH>(w3h + k + 64);
  };
  auto compute = [&](const uint4* v, int ch) {
    const size_t k = size_t(ch) * kChunk * 2;
#pragma unroll
    for (int G = 0; G < NG; ++G) {
      const uint4 x0 = ldg16(xr[G] + k), x1 = ldg16(xr[G] + k + 64);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t xb0 = word(x0, x1, 2 * j), xb1 = word(x0, x1, 2 * j + 1);
        mma16816(accg[G], word(v[0], v[1], 2 * j), word(v[2], v[3], 2 * j),
                 word(v[0], v[1], 2 * j + 1), word(v[2], v[3], 2 * j + 1), xb0, xb1);
        mma16816(accu[G], word(v[4], v[5], 2 * j), word(v[6], v[7], 2 * j),
                 word(v[4], v[5], 2 * j + 1), word(v[6], v[7], 2 * j + 1), xb0, xb1);
      }
    }
  };
  stream_chunks<DB>(warp % KS, nch, KS, load, compute);
#pragma unroll
  for (int G = 0; G < NG; ++G)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      red[((warp * kMaxNG + G) * 8 + i) * 32 + lane] = accg[G][i];
      red[((warp * kMaxNG + G) * 8 + 4 + i) * 32 + lane] = accu[G][i];
    }
  __syncthreads();
  // (row block, column group) pairs over the warps; slices added in order. Accumulator element
  // i: row g (i < 2) or g + 8, token column 2c + (i & 1)
  uint16_t* h = reinterpret_cast<uint16_t*>(a.h);
  for (int p = warp; p < RB * NG; p += kWarps) {
    const int rb = p / NG, G = p % NG;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float sg = 0.f, su = 0.f;
      for (int k = 0; k < KS; ++k) {
        const int w = rb * KS + k;
        sg += red[((w * kMaxNG + G) * 8 + i) * 32 + lane];
        su += red[((w * kMaxNG + G) * 8 + 4 + i) * 32 + lane];
      }
      const int j = G * 8 + 2 * c + (i & 1);
      if (j < n) {
        const int row = r0 + rb * kRows + g + (i >= 2 ? 8 : 0);
        if (lblk) {  // LoRA: + s B1 (A1 x), + s B3 (A3 x)
          const LoraOffsets lo = lora_offsets(a.d, a.w, a.lrank);
          const float* u = a.u13 + size_t(q0 + j) * 2 * a.lrank;
          sg += lora_up<__nv_bfloat16>(lblk, lo.b1, row, u, a.lrank, a.lscale);
          su += lora_up<__nv_bfloat16>(lblk, lo.b3, row, u + a.lrank, a.lrank, a.lscale);
        }
        h[size_t(q0 + j) * a.w + row] = f2bf(silu(sg) * su);
      }
    }
  }
  __syncthreads();
}

// GEMM2 for RB blocks of 32 output rows of W2 starting at r0 (two 16-row MMA tiles per warp that
// share the h fragments, so each lane keeps 8 weight loads in flight per chunk), contraction part
// kp of ks, and n <= 32 tokens; warp w owns row block w / KS and slice w % KS of the part (its
// chunks w % KS, w % KS + KS, ...).
// red: shared scratch [kWarps][kMaxNG][8][32] floats. Output plane kp of o.
template <int NG, bool DB, bool COH = false>
__device__ __forceinline__ void dec2_item(const FfnArgs& a, const char* blk, const void* lblk,
                                          int r0, int q0, int n, int kp, int ks, int RB, int KS,
                                          float* red) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const int rw = r0 + (warp / KS) * kRows2;
  const size_t rowb = size_t(a.w) * 2;
  const char* w2 = blk + size_t(2) * a.w * a.d * 2;
  const char* wg = w2 + size_t(rw + g) * rowb + c * 16;  // tile 0: rows g, g + 8
  const char* wh = wg + 8 * rowb;
  const char* vg = wg + 16 * rowb;                        // tile 1: rows 16 + g, 24 + g
  const char* vh = wg + 24 * rowb;
  const char* hr[NG];
#pragma unroll
  for (int G = 0; G < NG; ++G) {
    const int j = G * 8 + g;
    hr[G] = reinterpret_cast<const char*>(a.h) + size_t(q0 + (j < n ? j : 0)) * rowb + c * 16;
  }
  float acc[NG][8];
#pragma unroll
  for (int G = 0; G < NG; ++G)
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[G][i] = 0.f;

  int p0, p1;
  warp_slice(int(rowb / (kChunk * 2)), ks, kp, p0, p1);
  // one chunk's weights: tile 0 rows g / g+8 (lo, hi halves), then tile 1's
  auto load = [&](uint4* v, int ch) {
    const size_t k = size_t(ch) * kChunk * 2;
    v[0] = ldw16<COH>(wg + k); v[1] = ldw16<COH>(wg + k + 64);
    v[2] = ldw16<COH>(wh + k); v[3] = ldw16<COH>(wh + k + 64);
    v[4] = ldw16<COH>(vg + k); v[5] = ldw16<COH>(vg + k + 64);
    v[6] = ldw16<COH>(vh + k); v[7] = ldw16<COH>(vh + k + 64);
  };
  auto compute = [&](const uint4* v, int ch) {
    const size_t k = size_t(ch) * kChunk * 2;
#pragma unroll
    for (int G = 0; G < NG; ++G) {
      // h through L2 only: in the fused kernel other CTAs wrote it during this launch
      const uint4 x0 = ldcg16(hr[G] + k), x1 = ldcg16(hr[G] + k + 64);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t xb0 = word(x0, x1, 2 * j), xb1 = word(x0, x1, 2 * j + 1);
        mma16816(acc[G], word(v[0], v[1], 2 * j), word(v[2], v[3], 2 * j),
                 word(v[0], v[1], 2 * j + 1), word(v[2], v[3], 2 * j + 1), xb0, xb1);
        mma16816(acc[G] + 4, word(v[4], v[5], 2 * j), word(v[6], v[7], 2 * j),
                 word(v[4], v[5], 2 * j + 1), word(v[6], v[7], 2 * j + 1), xb0, xb1);
      }
    }
  };
  stream_chunks<DB>(p0 + warp % KS, p1, KS, load, compute);
#pragma unroll
  for (int G = 0; G < NG; ++G)
#pragma unroll
    for (int i = 0; i < 8; ++i) red[((warp * kMaxNG + G) * 8 + i) * 32 + lane] = acc[G][i];
  __syncthreads();
  // accumulator element i: tile i / 4, row g ((i & 3) < 2) or g + 8, token column 2c + (i & 1)
  float* o = a.o + size_t(kp) * a.o_plane;
  for (int p = warp; p < RB * NG; p += kWarps) {
    const int rb = p / NG, G = p % NG;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float sum = 0.f;
      for (int k = 0; k < KS; ++k) sum += red[(((rb * KS + k) * kMaxNG + G) * 8 + i) * 32 + lane];
      const int j = G * 8 + 2 * c + (i & 1);
      if (j < n) {
        const int row = r0 + rb * kRows2 + (i >> 2) * 16 + g + ((i & 3) >= 2 ? 8 : 0);
        if (lblk && kp == 0)  // LoRA: + s B2 (A2 h), once (in the first partial plane)
          sum += lora_up<__nv_bfloat16>(lblk, lora_offsets(a.d, a.w, a.lrank).b2, row,
                                        a.u2 + size_t(q0 + j) * a.lrank, a.lrank, a.lscale);
        o[size_t(q0 + j) * a.d + row] = sum;
      }
    }
  }
  __syncthreads();
}

// MAXNG: the largest token group (8 tokens each) this launch needs, from its batch size; a pass
// takes at most 8 * MAXNG tokens, and only the item variants up to MAXNG are compiled into the
// kernel, so the small-batch kernels keep the registers for double-buffered loads.
// One GEMM13 work item (RB blocks of 16 rows of one segment, all its tokens in passes of at most
// 8 * MAXNG); returns the segment.
template <int MAXNG, bool DBOK = true, bool COH = false>
__device__ __forceinline__ int run13_item(const FfnArgs& a, const DecItems& it, int item,
                                          float* red) {
  const int RB = it.rb, KS = kWarps / RB;
  const int p = dec_pos(it, item), s = it.seg[p];
  const int r0 = (item - it.first[p]) * kRows * RB;
  const char* blk = it.blk[s];
  const void* lblk = a.lrank ? a.lblk[s] : nullptr;
  // passes of at most 8 * MAXNG tokens; a later pass re-reads the rows from L2, not HBM
  for (int q0 = it.off[s]; q0 < it.off[s + 1]; q0 += 8 * MAXNG) {
    const int n = min(8 * MAXNG, it.off[s + 1] - q0);
    if (n <= 8) dec13_item<1, DBOK && MAXNG <= 2, COH>(a, blk, lblk, r0, q0, n, RB, KS, red);
    else if (MAXNG == 2 || n <= 16)
      dec13_item<(MAXNG >= 2 ? 2 : 1), false, COH>(a, blk, lblk, r0, q0, n, RB, KS, red);
    else dec13_item<MAXNG, false, COH>(a, blk, lblk, r0, q0, n, RB, KS, red);
  }
  return s;
}

// One GEMM2 work item (RB blocks of 32 rows of W2 of one segment, one contraction part).
template <int MAXNG, bool DBOK = true, bool COH = false>
__device__ __forceinline__ void run2_item(const FfnArgs& a, const DecItems& it, int item,
                                          float* red) {
  const int RB = it.rb, KS = kWarps / RB;
  const int p = dec_pos(it, item), s = it.seg[p];
  const int local = item - it.first[p];
  const int r0 = (local / it.ksplit) * kRows2 * RB, kp = local % it.ksplit;
  const char* blk = it.blk[s];
  const void* lblk = a.lrank ? a.lblk[s] : nullptr;
  for (int q0 = it.off[s]; q0 < it.off[s + 1]; q0 += 8 * MAXNG) {
    const int n = min(8 * MAXNG, it.off[s + 1] - q0);
    if (n <= 8)
      dec2_item<1, DBOK && MAXNG <= 2, COH>(a, blk, lblk, r0, q0, n, kp, it.ksplit, RB, KS, red);
    else if (MAXNG == 2 || n <= 16)
      dec2_item<(MAXNG >= 2 ? 2 : 1), false, COH>(a, blk, lblk, r0, q0, n, kp, it.ksplit, RB, KS,
                                                   red);
    else dec2_item<MAXNG, false, COH>(a, blk, lblk, r0, q0, n, kp, it.ksplit, RB, KS, red);
  }
}

template <int MAXNG>
__global__ void __launch_bounds__(kWarps * 32, 2) dec13_kernel(const __grid_constant__ FfnArgs a,
                                                               int RB) {
  pdl_wait();
  __shared__ DecItems it;
  __shared__ float red[kWarps * kMaxNG * 8 * 32];
  if (threadIdx.x < 32) build_dec_items(it, a, a.w, kRows, RB, 1);
  __syncthreads();
  for (int item = blockIdx.x; item < it.total; item += gridDim.x) run13_item<MAXNG>(a, it, item, red);
}

template <int MAXNG>
__global__ void __launch_bounds__(kWarps * 32, 2) dec2_kernel(const __grid_constant__ FfnArgs a,
                                                              int RB) {
  pdl_wait();
  __shared__ DecItems it;
  __shared__ float red[kWarps * kMaxNG * 8 * 32];
  if (threadIdx.x < 32) build_dec_items(it, a, a.d, kRows2, RB, a.ksplit);
  __syncthreads();
  for (int item = blockIdx.x; item < it.total; item += gridDim.x) run2_item<MAXNG>(a, it, item, red);
}

// the fused kernel holds both GEMMs' code, so it keeps double-buffered loads only where both fit
// the register budget without spills (see -Xptxas -v)
constexpr bool kFusedDB = false;

// Bounded wait (one thread) until segment s has `need` finished GEMM13 items; false (and the call
// aborted, so later waits return at once) if a.wait_ns pass (2 s unless a test shortened it) or
// the call is already aborting.
__device__ bool wait_segment(const FfnArgs& a, int s, int need) {
  const volatile int* p = a.done + s;
  const volatile int* abort = &a.hdr->abort;
  if (*p < need) {
    const uint64_t t0 = globaltimer_ns();
    while (*p < need) {
      if (*abort) return false;
      if (globaltimer_ns() - t0 > a.wait_ns) {
        set_error(a.err, kErrTimeout);
        const_cast<WsHeader*>(a.hdr)->abort = 1;
        return false;
      }
      __nanosleep(256);
    }
  }
  __threadfence();
  return true;
}

// Bounded wait (one thread) until every fetch piece of expert e's block that [off, off + len)
// touches carries this step's stamp, i.e. its bytes have landed; false (and the call aborted) if
// a.wait_ns pass or the call is already aborting.
__device__ bool wait_landed(const FfnArgs& a, unsigned epoch, int e, size_t off, size_t len) {
  const volatile unsigned* f = a.landed + size_t(e) * a.ppe;
  const volatile int* abort = &a.hdr->abort;
  const size_t p1 = (off + len - 1) / kFetchPiece;
  uint64_t t0 = 0;
  for (size_t p = off / kFetchPiece; p <= p1; ++p) {
    while (f[p] != epoch) {
      if (*abort) return false;
      const uint64_t now = globaltimer_ns();
      if (t0 == 0) t0 = now;
      else if (now - t0 > a.wait_ns) {
        set_error(a.err, kErrTimeout);
        const_cast<WsHeader*>(a.hdr)->abort = 1;
        return false;
      }
      __nanosleep(256);
    }
  }
  __threadfence();
  return true;
}

// GEMM13 and GEMM2 of a decode call in one launch. The work list is every GEMM13 item, then every
// GEMM2 item; CTAs claim items from a counter in the workspace (one atomic per item, issued for the
// next item while the current one runs), so CTAs that finish early take more and the launch ends
// when the work does, and CTAs that start late (an expert fetch kernel holding part of the SMs)
// only take what is left. A GEMM13 item publishes its segment's progress after its h rows are
// written and fenced; a GEMM2 item first waits (bounded) until its segment's GEMM13 items are all
// done, then reads h through L2. The waits always end: every GEMM13 item precedes every GEMM2 item
// in the claim order, so when a GEMM2 item is claimed its segment's GEMM13 items have all been
// claimed, each by a CTA that is running and finishes it without waiting on anything.
// A launch that fetches its own misses (a.nfetch > 0) first hands out fetcher roles from a
// counter the layer's cache step zeroed: the first a.nfetch CTAs to take a role copy the step's
// missed blocks from host memory piece by piece (pieces claimed from a second such counter, each
// stamped once written and fenced), before the grid-dependency wait (everything they read was
// written before the permutation began), then claim FFN items like the others. An item of a
// missed expert waits (bounded) for the stamps of the pieces it reads. Those waits end too: a CTA
// that holds an FFN item took its role after the a.nfetch fetchers took theirs, so every fetcher
// is running, and fetchers wait on nothing until all pieces are copied.
// FETCH: the build for launches that fetch their own misses (a.nfetch > 0); the plain build
// carries none of that code.
template <int MAXNG, bool FETCH>
__global__ void __launch_bounds__(kWarps * 32, 2)
    dec_fused_kernel(const __grid_constant__ FfnArgs a, int RB13, int RB2) {
  // fetching and streaming are compiled into the kernels of up to kStreamMaxT tokens (the host
  // only asks for them there)
  constexpr bool kStreams = FETCH && 8 * MAXNG <= kStreamMaxT;
  __shared__ DecItems it13, it2;
  __shared__ float red[kWarps * kMaxNG * 8 * 32];
  __shared__ int s_next, s_ok, s_role;
  const int warp = threadIdx.x >> 5;
  // Before the grid-dependency wait (the permutation lets this launch start while it runs), only
  // what was written before the permutation began is read: the segment block table (kernel
  // parameters, the cache's expert table) and, for the fetchers, the cache step's miss list, slot
  // addresses, step count and role and piece counters (zeroed by the cache step). So the copy of
  // the misses starts while the permutation still runs.
  fill_blk(it13, it2, a, 64);
  if constexpr (kStreams) {
    if (threadIdx.x == 64) s_role = int(atomicAdd(a.fctr, 1u));
  }
  __syncthreads();
  if constexpr (kStreams) {
    if (s_role < a.nfetch) {  // fetcher: copy the missed blocks' pieces until none are left
      const int nm = a.fmiss[0];  // copied even if the call aborts: the cache holds them now
      const size_t words = a.fbytes / 16, piece = kFetchPiece / 16;
      const int per = int((words + piece - 1) / piece);
      const unsigned epoch = static_cast<unsigned>(*a.epoch);
      for (;;) {
        if (threadIdx.x == 0) s_ok = int(atomicAdd(a.fctr + 1, 1u));
        __syncthreads();
        const int u = s_ok;
        __syncthreads();
        if (u >= nm * per) break;
        const int e = a.fmiss[1 + u / per];
        const size_t w0 = size_t(u % per) * piece, w1 = w0 + piece < words ? w0 + piece : words;
        copy_piece(reinterpret_cast<const uint4*>(a.fsrc[e]), reinterpret_cast<uint4*>(a.wtab[e]),
                   w0, w1);
        __threadfence();  // every thread's stores of the piece, before its stamp
        __syncthreads();
        if (threadIdx.x == 0)
          *reinterpret_cast<volatile unsigned*>(a.landed + size_t(e) * a.ppe + u % per) = epoch;
      }
    }
  }
  pdl_wait();
  if (warp == 0) build_dec_items(it13, a, a.w, kRows, RB13, 1, true);
  else if (warp == 1) build_dec_items(it2, a, a.d, kRows2, RB2, a.ksplit, true);
  else if (threadIdx.x == 64) {
    // the first claim goes out now, beside the work-list build (a fetcher only claims once the
    // pieces are all taken)
    s_next = atomicAdd(a.done + a.nseg + a.phase, 1);
  }
  __syncthreads();
  // Only the next claim stays live across an item body (the item index is consumed at its start;
  // the bounds are re-read from shared memory). Thread 0 issues the claim before the body and
  // publishes it after, so the atomic's round trip overlaps warp 0's weight loads.
  for (;;) {
    const int item = s_next;
    __syncthreads();  // every thread has read it before thread 0 publishes the next
    if (item < 0 || item >= it13.total + it2.total) break;
    int next = 0;
    if (threadIdx.x == 0) next = atomicAdd(a.done + a.nseg + a.phase, 1);
    if (item < it13.total) {
      if (!a.withhold13) {  // (a test withholds GEMM13 items to make the GEMM2 waits run out)
        const int p = dec_pos(it13, item), s = it13.seg[p];
        const bool streamed = kStreams && seg_streamed(a, s, it13.stream);
        int ok = 1;
        if (streamed) {  // the item's rows of W1 and of W3 must have landed
          if (threadIdx.x == 0) {
            const size_t rowb = size_t(a.d) * 2, r0 = size_t(item - it13.first[p]) * kRows * it13.rb;
            const size_t n = size_t(kRows) * it13.rb * rowb;
            s_ok = wait_landed(a, it13.epoch, s, r0 * rowb, n) &&
                   wait_landed(a, it13.epoch, s, (a.w + r0) * rowb, n);
          }
          __syncthreads();
          ok = s_ok;
        }
        if (ok) {
          if constexpr (kStreams) {
            if (streamed) run13_item<MAXNG, kFusedDB, true>(a, it13, item, red);
            else run13_item<MAXNG, kFusedDB>(a, it13, item, red);
          } else {
            run13_item<MAXNG, kFusedDB>(a, it13, item, red);
          }
          __threadfence();  // this CTA's h rows, before the segment's count moves
          __syncthreads();
          if (threadIdx.x == 0) atomicAdd(a.done + s, 1);
        }
      }
    } else {
      const int i2 = item - it13.total;
      const int p = dec_pos(it2, i2), s = it2.seg[p];
      const bool streamed = kStreams && seg_streamed(a, s, it2.stream);
      // every segment with work has w / (16 rb) GEMM13 items; a streamed segment's item also
      // waits for its rows of W2
      if (threadIdx.x == 0) {
        bool ok = wait_segment(a, s, a.w / (kRows * it13.rb));
        if (ok && streamed) {
          const size_t rowb = size_t(a.w) * 2;
          const size_t r0 = size_t((i2 - it2.first[p]) / it2.ksplit) * kRows2 * it2.rb;
          ok = wait_landed(a, it2.epoch, s, size_t(2) * a.w * a.d * 2 + r0 * rowb,
                           size_t(kRows2) * it2.rb * rowb);
        }
        s_ok = ok ? 1 : 0;
      }
      __syncthreads();
      if (s_ok) {
        if constexpr (kStreams) {
          if (streamed) run2_item<MAXNG, kFusedDB, true>(a, it2, i2, red);
          else run2_item<MAXNG, kFusedDB>(a, it2, i2, red);
        } else {
          run2_item<MAXNG, kFusedDB>(a, it2, i2, red);
        }
      }
    }
    if (threadIdx.x == 0) s_next = next;
    __syncthreads();
  }
}

int blocks_per_sm(const void* fn) {
  int nb = 1;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, fn, kWarps * 32, 0) != cudaSuccess || nb < 1)
    nb = 1;
  return nb;
}

}  // namespace

int decode_ksplit(int T) { return T <= 4 ? 8 : (T <= 16 ? 2 : 1); }

// Row blocks per CTA item: the smallest RB in {1, 2, 4, 8} whose 8 / RB contraction slices give
// every warp at least min_chunks chunks of 64 (while the rows still split into whole items). More
// slices mean finer items and better balance; fewer mean longer, better pipelined loops.
// At up to 4 tokens a launch is latency-bound (few items per CTA, each warp's chunks in series),
// so GEMM13 items take half the minimum (finer items, each warp walking fewer chunks); beyond
// that the longer loops pay. A function of the layer and the batch only, like every item shape.
constexpr int kMinChunks = 8;
constexpr int kMinChunksSmallBatch = 4;
int rows_per_item(int rows, int contraction, int rows_per_warp, int min_chunks = kMinChunks) {
  const int nch = contraction / kChunk;
  int rb = 1;
  while (rb < kWarps && nch / (kWarps / rb) < min_chunks && rows % (rows_per_warp * rb * 2) == 0)
    rb *= 2;
  return rb;
}

template <int MAXNG>
cudaError_t launch_decode_ng(const FfnArgs& a, int num_sms, cudaStream_t s, int stages,
                             int reserved) {
  static const int nb13 = blocks_per_sm(reinterpret_cast<const void*>(dec13_kernel<MAXNG>));
  static const int nb2 = blocks_per_sm(reinterpret_cast<const void*>(dec2_kernel<MAXNG>));
  // one CTA per SM slot, less the slots left to another kernel
  const int g13 = max(num_sms, num_sms * nb13 - reserved);
  const int g2 = max(num_sms, num_sms * nb2 - reserved);
  const int rb13 = rows_per_item(a.w, a.d, kRows, a.T <= 4 ? kMinChunksSmallBatch : kMinChunks);
  const int rb2 = rows_per_item(a.d, a.w / a.ksplit, kRows2);
  cudaError_t e = cudaSuccess;
  if (stages == 3 && a.done && a.lrank == 0) {
    // both GEMMs in one launch with claimed items
    static const int nbf =
        blocks_per_sm(reinterpret_cast<const void*>(dec_fused_kernel<MAXNG, false>));
    const int gf = max(num_sms, num_sms * nbf - reserved);
    if constexpr (8 * MAXNG <= kStreamMaxT) {
      if (a.nfetch > 0) {  // fetching its own misses
        prof_begin(kProfDecFetch, s);
        e = launch_pdl(dec_fused_kernel<MAXNG, true>, dim3(gf), dim3(kWarps * 32), 0, s, a, rb13,
                       rb2);
        prof_end(kProfDecFetch, s);
        return e != cudaSuccess ? e : cudaGetLastError();
      }
    }
    prof_begin(kProfDecFused, s);
    e = launch_pdl(dec_fused_kernel<MAXNG, false>, dim3(gf), dim3(kWarps * 32), 0, s, a, rb13, rb2);
    prof_end(kProfDecFused, s);
    return e != cudaSuccess ? e : cudaGetLastError();
  }
  if (stages & 1) {
    prof_begin(kProfDec13, s);
    e = launch_pdl(dec13_kernel<MAXNG>, dim3(g13), dim3(kWarps * 32), 0, s, a, rb13);
    prof_end(kProfDec13, s);
    if (e == cudaSuccess) e = cudaGetLastError();
  }
  if (e != cudaSuccess || !(stages & 2)) return e;
  prof_begin(kProfDec2, s);
  e = launch_pdl(dec2_kernel<MAXNG>, dim3(g2), dim3(kWarps * 32), 0, s, a, rb2);
  prof_end(kProfDec2, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_ffn_decode(const FfnArgs& args, int num_sms, cudaStream_t s, int stages,
                              int reserved) {
  FfnArgs a = args;
  a.wait_ns = test_wait_limit_ns();
  a.withhold13 = test_withhold_gemm13() ? 1 : 0;
  // a segment holds at most T tokens (routed experts: distinct per token; shared: all T)
  if (a.T <= 8) return launch_decode_ng<1>(a, num_sms, s, stages, reserved);
  if (a.T <= 16) return launch_decode_ng<2>(a, num_sms, s, stages, reserved);
  return launch_decode_ng<4>(a, num_sms, s, stages, reserved);
}

}  // namespace mcft
