// encode.cu -- re-encoding of the draft string into target tokens (§4.2,
// App. A.1), the Lemma-1 byte check (App. A.1) and the delta-pos histogram of
// the DTW paths (§4.1, App. K).
//
// Re-encoding is greedy longest match over the target vocabulary, through an
// index of every prefix of every token: an open-addressing table whose slot
// holds the prefix's key, its length and the token it spells exactly (if any).
// Walking the prefixes of the text at position p one byte at a time, the walk
// stops at the first prefix no token starts with, so a lookup costs about as
// many probes as the match is long. One warp per request; a second kernel (one
// CTA) turns the per-request counts into CSR offsets, a third compacts the
// tokens (one warp per request).
#include <cstdint>
#include <cstring>
#include <vector>

#include "tt_device.cuh"
#include "tt_launch.h"

namespace tt {

namespace {

// ------------------------------------------------------------- the index

struct IndexHeader {
  uint32_t magic;
  int32_t n_slots;   // power of two
  int32_t max_len;   // longest token in bytes
  int32_t n_tokens;
  int64_t reserved[6];
};

struct Slot {
  uint64_t key;  // the prefix's bytes (up to 8) or its fingerprint (longer)
  int32_t len;   // prefix length in bytes; 0 = empty slot
  int32_t id;    // token spelled by exactly this prefix, -1 = none
};

static_assert(sizeof(IndexHeader) == 64 && sizeof(Slot) == 16, "index layout");
constexpr uint32_t kIndexMagic = 0x58495454u;
constexpr int kMaxIndexTokens = 1 << 22;  // ids fit 22 bits beside a 9-bit length

// MurmurHash3's 64-bit finaliser (A. Appleby, public domain).
__host__ __device__ __forceinline__ uint64_t fmix64(uint64_t x) {
  x ^= x >> 33;
  x *= 0xff51afd7ed558ccdull;
  x ^= x >> 33;
  x *= 0xc4ceb9fe1a85ec53ull;
  x ^= x >> 33;
  return x;
}

// Key of a prefix of length L from the key of its first L-1 bytes: the bytes
// themselves (little-endian) up to 8, then a chained fingerprint.
__host__ __device__ __forceinline__ uint64_t key_step(uint64_t key, uint8_t byte, int L) {
  if (L <= 8) return key | (uint64_t(byte) << (8 * (L - 1)));
  return fmix64(key + uint64_t(byte) * 0x9e3779b97f4a7c15ull + uint64_t(L));
}

__host__ __device__ __forceinline__ uint32_t home_slot(uint64_t key, int L, int n_slots) {
  return uint32_t(fmix64(key ^ (uint64_t(L) * 0xc2b2ae3d27d4eb4full))) & uint32_t(n_slots - 1);
}

size_t slots_for(int64_t n_bytes) {
  const size_t need = size_t(2 * (n_bytes > 0 ? n_bytes : 1));
  size_t s = 16;
  while (s < need) s <<= 1;
  return s;
}

// ------------------------------------------------------------- re-encoding

constexpr int kEncWarps = 4;

struct EncArgs {
  int B, n_draft, max_m;
  const int32_t* draft_off;
  const int32_t* draft_ids;
  tt_vocab vd, vt;
  const IndexHeader* hdr;
  const Slot* slots;
  int32_t* pad_ids;  // [B * max_m]
  int32_t* counts;   // [B]
  int32_t* status;   // [B]
};

__device__ __forceinline__ int64_t warp_sum_i64(int64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ bool token_ok(const tt_vocab& v, int id) {
  if (id < 0 || id >= v.n_tokens) return false;
  const int64_t o0 = v.offsets[id], o1 = v.offsets[id + 1];
  return o0 >= 0 && o1 >= o0 && o1 <= v.n_bytes;
}

// Token `id` of vt spells s[0..L).
__device__ bool spells(const tt_vocab& vt, int id, const uint8_t* s, int L) {
  const int64_t o0 = vt.offsets[id];
  if (vt.offsets[id + 1] - o0 != L) return false;
  for (int x = 0; x < L; ++x)
    if (vt.bytes[o0 + x] != s[x]) return false;
  return true;
}

__global__ void __launch_bounds__(32 * kEncWarps) encode_kernel(EncArgs a) {
  __shared__ uint8_t s_text[kEncWarps][TT_MAX_ENCODE_BYTES];
  // longest match at each position: (token id << 9) | length, 0 = none
  __shared__ int32_t s_match[kEncWarps][TT_MAX_ENCODE_BYTES];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * kEncWarps + warp;
  if (b >= a.B) return;
  uint8_t* text = s_text[warp];
  int32_t* match = s_match[warp];

  int st = 0, k = 0, d0 = 0, m = 0;
  const bool index_ok = a.hdr->magic == kIndexMagic && a.hdr->n_slots >= 16 &&
                        (a.hdr->n_slots & (a.hdr->n_slots - 1)) == 0;
  if (!csr_ok(a.draft_off, b, a.n_draft)) {
    st = TT_REQ_BAD_OFFSETS;
  } else {
    d0 = a.draft_off[b];
    k = a.draft_off[b + 1] - d0;
    if (k == 0) st |= TT_REQ_EMPTY;
  }
  int n = 0;
  if (st == 0) {
    int bad = 0;
    int64_t tot = 0;
    for (int i = lane; i < k; i += 32) {
      const int id = a.draft_ids[d0 + i];
      if (!token_ok(a.vd, id)) {
        bad = 1;
        continue;
      }
      tot += a.vd.offsets[id + 1] - a.vd.offsets[id];
    }
    tot = warp_sum_i64(tot);
    if (__any_sync(0xffffffffu, bad)) st |= TT_REQ_ID_OUT_OF_RANGE;
    else if (tot > TT_MAX_ENCODE_BYTES) st |= TT_REQ_TOO_LONG;
    n = int(tot);
  }
  if (st == 0 && !index_ok) st = TT_REQ_INTERNAL;
  if (st == 0) {
    // decode_d: the draft tokens' bytes, 32 tokens per round
    int base = 0;
    for (int r = 0; r < k; r += 32) {
      const int i = r + lane;
      int len = 0;
      int64_t o0 = 0;
      if (i < k) {
        const int id = a.draft_ids[d0 + i];
        o0 = a.vd.offsets[id];
        len = int(a.vd.offsets[id + 1] - o0);
      }
      int incl = len;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      const int start = base + incl - len;
      for (int x = 0; x < len; ++x) text[start + x] = a.vd.bytes[o0 + x];
      base += __shfl_sync(0xffffffffu, incl, 31);
    }
    __syncwarp();
    // the longest target token at every position
    const int max_len = a.hdr->max_len, n_slots = a.hdr->n_slots;
    for (int p = lane; p < n; p += 32) {
      uint64_t key = 0;
      int best = 0;
      const int lim = min(max_len, n - p);
      for (int L = 1; L <= lim; ++L) {
        key = key_step(key, text[p + L - 1], L);
        uint32_t s = home_slot(key, L, n_slots);
        int found = -2;  // -2: no token starts with these L bytes
        for (int probe = 0; probe < n_slots; ++probe) {  // the table is at most half full
          const Slot sl = a.slots[s];
          if (sl.len == 0) break;
          if (sl.len == L && sl.key == key) {
            found = sl.id;
            break;
          }
          s = (s + 1) & uint32_t(n_slots - 1);
        }
        if (found == -2) break;
        // (an id past vt's table means the index belongs to another vocabulary)
        if (found >= 0 && found < a.vt.n_tokens && (L <= 8 || spells(a.vt, found, text + p, L)))
          best = (found << 9) | L;
      }
      match[p] = best;
    }
    __syncwarp();
    // encode_t: greedy walk over the matches
    if (lane == 0) {
      int p = 0;
      while (p < n) {
        const int mt = match[p];
        if (mt == 0) {
          st |= TT_REQ_NO_MATCH;
          break;
        }
        if (m >= a.max_m) {
          st |= TT_REQ_TOO_LONG;
          break;
        }
        a.pad_ids[int64_t(b) * a.max_m + m] = mt >> 9;
        ++m;
        p += mt & 511;
      }
    }
  }
  if (lane == 0) {
    a.counts[b] = st == 0 ? m : 0;
    a.status[b] = st;
  }
}

struct FinArgs {
  int B, max_m, capacity;
  const int32_t* pad_ids;
  const int32_t* counts;
  int32_t* status;
  int32_t* target_off;
  int32_t* target_ids;
};

constexpr int kFinThreads = 1024;

// Inclusive block scan of one int64 per thread; returns the block total in *total.
__device__ int64_t block_scan(int64_t v, int64_t* s_warp, int64_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  if (lane == 31) s_warp[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int64_t w = lane < kFinThreads / 32 ? s_warp[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t n = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += n;
    }
    s_warp[lane] = w;  // inclusive over warps
  }
  __syncthreads();
  const int64_t before = warp > 0 ? s_warp[warp - 1] : 0;
  *total = s_warp[kFinThreads / 32 - 1];
  __syncthreads();
  return v + before;
}

// One CTA: CSR offsets with the capacity rule.
__global__ void __launch_bounds__(kFinThreads) encode_finish_kernel(FinArgs a) {
  __shared__ int64_t s_warp[kFinThreads / 32];
  int64_t carry_all = 0, carry_written = 0;
  if (threadIdx.x == 0) a.target_off[0] = 0;
  for (int c = 0; c < a.B; c += kFinThreads) {
    const int b = c + threadIdx.x;
    const int cnt = b < a.B ? a.counts[b] : 0;
    int64_t tot;
    const int64_t end_all = carry_all + block_scan(cnt, s_warp, &tot);
    carry_all += tot;
    int st = b < a.B ? a.status[b] : 1;
    int written = cnt;
    if (st == 0 && end_all > a.capacity) {
      st |= TT_REQ_TOO_LONG;
      written = 0;
    }
    const int64_t end_w = carry_written + block_scan(written, s_warp, &tot);
    carry_written += tot;
    if (b < a.B) {
      a.status[b] = st;
      a.target_off[b + 1] = int32_t(end_w);
    }
  }
}

constexpr int kCompactWarps = 8;

// Compaction of the padded tokens into the CSR output: one warp per request.
__global__ void __launch_bounds__(32 * kCompactWarps) encode_compact_kernel(FinArgs a) {
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * kCompactWarps + (threadIdx.x >> 5);
  if (b >= a.B) return;
  const int o0 = a.target_off[b], n = a.target_off[b + 1] - o0;
  for (int j = lane; j < n; j += 32) a.target_ids[o0 + j] = a.pad_ids[int64_t(b) * a.max_m + j];
}

// ------------------------------------------------------- Lemma-1 byte check

constexpr int kConsWarps = 4;

struct ConsArgs {
  int B, n_draft, n_target, max_k, max_m;
  const int32_t* draft_off;
  const int32_t* draft_ids;
  const int32_t* target_off;
  const int32_t* target_ids;
  tt_vocab vd, vt;
  int32_t* status;
};

// Inclusive prefix sums of the byte lengths of n tokens into pre[1..n] (pre[0] = 0).
__device__ void byte_prefix(const tt_vocab& v, const int32_t* ids, int n, int32_t* pre, int lane) {
  int base = 0;
  if (lane == 0) pre[0] = 0;
  for (int r = 0; r < n; r += 32) {
    const int i = r + lane;
    const int len = i < n ? int(v.offsets[ids[i] + 1] - v.offsets[ids[i]]) : 0;
    int incl = len;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int x = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += x;
    }
    if (i < n) pre[i + 1] = base + incl;
    base += __shfl_sync(0xffffffffu, incl, 31);
  }
  __syncwarp();
}

// Byte at position p of the concatenation (pre: prefix sums of n tokens).
__device__ __forceinline__ uint8_t byte_at(const tt_vocab& v, const int32_t* ids,
                                           const int32_t* pre, int n, int p) {
  int lo = 0, hi = n - 1;  // last token whose start is <= p
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (pre[mid] <= p) lo = mid;
    else hi = mid - 1;
  }
  return v.bytes[v.offsets[ids[lo]] + (p - pre[lo])];
}

__global__ void __launch_bounds__(32 * kConsWarps) consistency_kernel(ConsArgs a) {
  __shared__ int32_t s_pd[kConsWarps][TT_MAX_K + 1];
  __shared__ int32_t s_pt[kConsWarps][TT_MAX_M + 1];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * kConsWarps + warp;
  if (b >= a.B) return;
  int st = 0;
  if (!csr_ok(a.draft_off, b, a.n_draft) || !csr_ok(a.target_off, b, a.n_target)) {
    if (lane == 0) a.status[b] = TT_REQ_BAD_OFFSETS;
    return;
  }
  const int d0 = a.draft_off[b], k = a.draft_off[b + 1] - d0;
  const int t0 = a.target_off[b], m = a.target_off[b + 1] - t0;
  if (k > a.max_k || m > a.max_m) st |= TT_REQ_TOO_LONG;
  int bad = 0;
  for (int i = lane; i < k; i += 32) bad |= !token_ok(a.vd, a.draft_ids[d0 + i]);
  for (int j = lane; j < m; j += 32) bad |= !token_ok(a.vt, a.target_ids[t0 + j]);
  if (__any_sync(0xffffffffu, bad)) st |= TT_REQ_ID_OUT_OF_RANGE;
  if (st == 0) {
    const int32_t* D = a.draft_ids + d0;
    const int32_t* T = a.target_ids + t0;
    byte_prefix(a.vd, D, k, s_pd[warp], lane);
    byte_prefix(a.vt, T, m, s_pt[warp], lane);
    const int nd = s_pd[warp][k], nt = s_pt[warp][m];
    int diff = nd != nt;
    for (int p = lane; !diff && p < nd; p += 32)
      diff = byte_at(a.vd, D, s_pd[warp], k, p) != byte_at(a.vt, T, s_pt[warp], m, p);
    if (__any_sync(0xffffffffu, diff)) st |= TT_REQ_INCONSISTENT;
  }
  if (lane == 0) a.status[b] = st;
}

// --------------------------------------------------- delta-pos histogram

constexpr int kDposWarps = 4;

struct DposArgs {
  int B, n_draft, n_target, mode, n_bins;
  const int32_t* draft_off;
  const int32_t* target_off;
  const int32_t* path;
  const int32_t* path_len;
  const int32_t* map;
  unsigned long long* hist;
};

__global__ void __launch_bounds__(32 * kDposWarps) dpos_kernel(DposArgs a) {
  __shared__ unsigned int s_hist[TT_MAX_DPOS_BINS];
  for (int x = threadIdx.x; x < a.n_bins; x += blockDim.x) s_hist[x] = 0;
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int top = a.n_bins - 1;
  for (int b = blockIdx.x * kDposWarps + warp; b < a.B; b += gridDim.x * kDposWarps) {
    if (!csr_ok(a.draft_off, b, a.n_draft) || !csr_ok(a.target_off, b, a.n_target)) continue;
    const int d0 = a.draft_off[b], k = a.draft_off[b + 1] - d0;
    const int t0 = a.target_off[b], m = a.target_off[b + 1] - t0;
    const int len = min(a.path_len[b], k + m);  // the request's path capacity
    if (len <= 0) continue;
    if (a.mode == 0) {
      const int32_t* pp = a.path + 2 * (int64_t(d0) + t0);
      for (int x = lane; x < len; x += 32) {
        const int d = abs(pp[2 * x] - pp[2 * x + 1]);
        atomicAdd(&s_hist[min(d, top)], 1u);
      }
    } else {
      for (int j = lane; j < m; j += 32) {
        const int d = abs(a.map[t0 + j] - j);
        atomicAdd(&s_hist[min(d, top)], 1u);
      }
    }
  }
  __syncthreads();
  for (int x = threadIdx.x; x < a.n_bins; x += blockDim.x)
    if (s_hist[x]) atomicAdd(&a.hist[x], (unsigned long long)s_hist[x]);
}

bool batch_ok_lite(const tt_batch* b) {
  if (!b || b->B < 0 || b->n_draft < 0 || b->n_target < 0) return false;
  if (b->B == 0) return true;
  return b->draft_off && b->target_off && b->max_k >= 1 && b->max_k <= TT_MAX_K &&
         b->max_m >= 1 && b->max_m <= TT_MAX_M;
}

bool vocab_ok_lite(const tt_vocab* v) {
  return v && v->bytes && v->offsets && v->n_tokens >= 1 && v->n_bytes >= 0;
}

}  // namespace
}  // namespace tt

using namespace tt;

extern "C" size_t tt_vocab_index_bytes(int32_t n_tokens, int64_t n_bytes) {
  (void)n_tokens;
  return sizeof(IndexHeader) + slots_for(n_bytes) * sizeof(Slot);
}

extern "C" tt_status tt_vocab_index_build(const uint8_t* bytes, const int64_t* offsets,
                                          int32_t n_tokens, void* index, size_t index_bytes) {
  if (!offsets || !index || n_tokens < 1 || n_tokens > kMaxIndexTokens) return TT_ERR_INVALID_ARG;
  int64_t total = 0, max_len = 0;
  for (int32_t v = 0; v < n_tokens; ++v) {
    const int64_t len = offsets[v + 1] - offsets[v];
    if (offsets[v] < 0 || len < 0) return TT_ERR_INVALID_ARG;
    if (len > TT_MAX_TOKEN_BYTES) return TT_ERR_UNSUPPORTED;
    total += len;
    if (len > max_len) max_len = len;
  }
  if (total > 0 && !bytes) return TT_ERR_INVALID_ARG;
  if (index_bytes < sizeof(IndexHeader) + 16 * sizeof(Slot)) return TT_ERR_INVALID_ARG;
  size_t n_slots = 16;
  while (n_slots * 2 * sizeof(Slot) + sizeof(IndexHeader) <= index_bytes) n_slots *= 2;
  if (n_slots < size_t(2 * total) || n_slots > (size_t(1) << 30)) return TT_ERR_INVALID_ARG;

  IndexHeader* hdr = static_cast<IndexHeader*>(index);
  Slot* slots = reinterpret_cast<Slot*>(static_cast<char*>(index) + sizeof(IndexHeader));
  std::memset(index, 0, sizeof(IndexHeader) + n_slots * sizeof(Slot));
  std::vector<int32_t> owner(n_slots, -1);  // a token whose prefix created the slot
  const uint32_t mask = uint32_t(n_slots - 1);
  for (int32_t v = 0; v < n_tokens; ++v) {  // in id order: the smallest id keeps a string
    const uint8_t* s = bytes + offsets[v];
    const int len = int(offsets[v + 1] - offsets[v]);
    uint64_t key = 0;
    for (int L = 1; L <= len; ++L) {
      key = key_step(key, s[L - 1], L);
      uint32_t h = home_slot(key, L, int(n_slots));
      for (;;) {
        Slot& sl = slots[h];
        if (sl.len == 0) {
          sl.key = key;
          sl.len = L;
          sl.id = L == len ? v : -1;
          owner[h] = v;
          break;
        }
        if (sl.len == L && sl.key == key) {
          if (L > 8 && std::memcmp(bytes + offsets[owner[h]], s, size_t(L)) != 0)
            return TT_ERR_UNSUPPORTED;  // two different prefixes share a fingerprint
          if (L == len && sl.id < 0) sl.id = v;
          break;
        }
        h = (h + 1) & mask;
      }
    }
  }
  hdr->magic = kIndexMagic;
  hdr->n_slots = int32_t(n_slots);
  hdr->max_len = int32_t(max_len);
  hdr->n_tokens = n_tokens;
  return TT_OK;
}

extern "C" size_t tt_encode_workspace_bytes(int32_t B, int32_t max_m) {
  if (B < 0 || max_m < 0) return 0;
  return align256(sizeof(int32_t) * size_t(B) * size_t(max_m)) +
         align256(sizeof(int32_t) * size_t(B > 0 ? B : 1));
}

extern "C" tt_status tt_encode(int32_t B, int32_t n_draft, const int32_t* draft_off,
                               const int32_t* draft_ids,
                               const tt_vocab* vd, const tt_vocab* vt, const void* vt_index,
                               int32_t max_m, int32_t capacity, int32_t* target_off,
                               int32_t* target_ids, int32_t* status, void* workspace,
                               size_t workspace_bytes, void* stream) {
  if (B < 0 || n_draft < 0 || !target_off || max_m < 1 || max_m > TT_MAX_M || capacity < 0)
    return TT_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (B == 0) {
    const cudaError_t e = cudaMemsetAsync(target_off, 0, sizeof(int32_t), s);
    return e == cudaSuccess ? TT_OK : record_cuda_error(e);
  }
  if (!draft_off || (n_draft > 0 && !draft_ids) || !status || !vt_index ||
      (capacity > 0 && !target_ids) ||
      !vocab_ok_lite(vd) || !vocab_ok_lite(vt))
    return TT_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(vt_index) & 15) != 0) return TT_ERR_INVALID_ARG;
  if (!workspace || workspace_bytes < tt_encode_workspace_bytes(B, max_m) ||
      (reinterpret_cast<uintptr_t>(workspace) & 255) != 0)
    return TT_ERR_INVALID_ARG;
  EncArgs a;
  a.B = B;
  a.n_draft = n_draft;
  a.max_m = max_m;
  a.draft_off = draft_off;
  a.draft_ids = draft_ids;
  a.vd = *vd;
  a.vt = *vt;
  a.hdr = static_cast<const IndexHeader*>(vt_index);
  a.slots = reinterpret_cast<const Slot*>(static_cast<const char*>(vt_index) + sizeof(IndexHeader));
  a.pad_ids = static_cast<int32_t*>(workspace);
  a.counts = reinterpret_cast<int32_t*>(static_cast<char*>(workspace) +
                                        align256(sizeof(int32_t) * size_t(B) * size_t(max_m)));
  a.status = status;
  encode_kernel<<<(B + kEncWarps - 1) / kEncWarps, 32 * kEncWarps, 0, s>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return record_cuda_error(e);
  FinArgs f;
  f.B = B;
  f.max_m = max_m;
  f.capacity = capacity;
  f.pad_ids = a.pad_ids;
  f.counts = a.counts;
  f.status = status;
  f.target_off = target_off;
  f.target_ids = target_ids;
  encode_finish_kernel<<<1, kFinThreads, 0, s>>>(f);
  if ((e = cudaGetLastError()) != cudaSuccess) return record_cuda_error(e);
  encode_compact_kernel<<<(B + kCompactWarps - 1) / kCompactWarps, 32 * kCompactWarps, 0, s>>>(f);
  e = cudaGetLastError();
  return e == cudaSuccess ? TT_OK : record_cuda_error(e);
}

extern "C" tt_status tt_consistency(const tt_batch* batch, const tt_vocab* vd, const tt_vocab* vt,
                                    int32_t* status, void* stream) {
  if (!batch_ok_lite(batch)) return TT_ERR_INVALID_ARG;
  if (batch->B == 0) return TT_OK;
  if (!status || !vocab_ok_lite(vd) || !vocab_ok_lite(vt) ||
      (batch->n_draft > 0 && !batch->draft_ids) || (batch->n_target > 0 && !batch->target_ids))
    return TT_ERR_INVALID_ARG;
  ConsArgs a;
  a.B = batch->B;
  a.n_draft = batch->n_draft;
  a.n_target = batch->n_target;
  a.max_k = batch->max_k;
  a.max_m = batch->max_m;
  a.draft_off = batch->draft_off;
  a.draft_ids = batch->draft_ids;
  a.target_off = batch->target_off;
  a.target_ids = batch->target_ids;
  a.vd = *vd;
  a.vt = *vt;
  a.status = status;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  consistency_kernel<<<(a.B + kConsWarps - 1) / kConsWarps, 32 * kConsWarps, 0, s>>>(a);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? TT_OK : record_cuda_error(e);
}

extern "C" tt_status tt_dpos_hist(const tt_batch* batch, const int32_t* path,
                                  const int32_t* path_len, const int32_t* map, int32_t mode,
                                  int32_t n_bins, int64_t* hist, void* stream) {
  if (!batch_ok_lite(batch) || (mode != 0 && mode != 1) || n_bins < 1 ||
      n_bins > TT_MAX_DPOS_BINS || !hist)
    return TT_ERR_INVALID_ARG;
  if (batch->B == 0) return TT_OK;
  if (!path_len || (mode == 0 && !path) || (mode == 1 && batch->n_target > 0 && !map))
    return TT_ERR_INVALID_ARG;
  DposArgs a;
  a.B = batch->B;
  a.n_draft = batch->n_draft;
  a.n_target = batch->n_target;
  a.mode = mode;
  a.n_bins = n_bins;
  a.draft_off = batch->draft_off;
  a.target_off = batch->target_off;
  a.path = path;
  a.path_len = path_len;
  a.map = map;
  a.hist = reinterpret_cast<unsigned long long*>(hist);
  int dev = 0, sms = 148;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int want = (a.B + kDposWarps - 1) / kDposWarps;
  const int grid = want < 2 * sms ? want : 2 * sms;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  dpos_kernel<<<grid, 32 * kDposWarps, 0, s>>>(a);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? TT_OK : record_cuda_error(e);
}
