// align.cu -- Dynamic Token Warping between draft and proxy target tokens
// (§4.1, Alg. 1) with the byte-level Levenshtein token distance (App. H).
//
// One warp per request (sequence pair), several pairs per CTA, each warp
// looping over pairs when the grid is smaller than the batch. Per pair:
//  1. stage the tokens' byte strings in shared memory (packed 8-byte words);
//  2. fill the banded local-cost tile d(i,j), one byte per cell, with all 32
//     lanes (two interleaved bit-parallel edit distances per lane for tokens
//     of <= 8 bytes, a plain DP otherwise);
//  3. sweep the anti-diagonals i + j = s: every cell of a diagonal depends
//     only on the two previous diagonals, kept in registers (one cell per
//     lane, neighbours by shuffles) while the band's half-width is at most
//     31, else in three rotating shared buffers; each cell's choice of
//     predecessor overwrites its cost in the tile (diagonal, then (i-1,j),
//     then (i,j-1) on ties);
//  4. backtrack from (k, m) on one lane, then write path, C*, the map
//     i*(j) = max{i : (i,j) on the path} and the needed-draft-row flags.
#include <algorithm>
#include <cstdint>

#include "tt_device.cuh"
#include "tt_launch.h"

namespace tt {

namespace {

// Bit i set iff byte i of the packed string P equals c. Each half's bytes of
// P ^ c...c are tested for zero exactly (the high bit of a byte of
// ~(((t & 0x7f..) + 0x7f..) | t | 0x7f..) is set iff the byte of t is 0); the
// eight flags, at bits 8y (low half) and 8y + 4 (high half) after the shifts,
// are gathered into bits 0..7 by one multiply: the multiplier's bits 7, 14,
// 21, 28 send flag bit q to q + 7 .. q + 28, and each product bit receives at
// most one term (the flags lie 4 apart, the shifts differ mod 4), so nothing
// carries and bits 28..35 hold the flags in byte order.
__device__ __forceinline__ uint32_t eq_mask8(uint64_t P, uint32_t c) {
  const uint32_t cc = c * 0x01010101u;
  const uint32_t tl = uint32_t(P) ^ cc, th = uint32_t(P >> 32) ^ cc;
  const uint32_t zl = ~(((tl & 0x7f7f7f7fu) + 0x7f7f7f7fu) | tl | 0x7f7f7f7fu);
  const uint32_t zh = ~(((th & 0x7f7f7f7fu) + 0x7f7f7f7fu) | th | 0x7f7f7f7fu);
  const uint32_t f = (zl >> 7) | (zh >> 3);
  return uint32_t((uint64_t(f) * 0x10204080ull) >> 28) & 0xFFu;
}

// Edit distance of two byte strings of at most 8 bytes, packed little-endian,
// by the bit-parallel column recurrence of Myers (1999) in Hyyro's form for
// global distance: one pass over the text, one 8-bit vector per column.
__device__ __forceinline__ int lev_packed8(uint64_t P, int lp, uint64_t T, int lt) {
  if (lp == 0) return lt;
  if (lt == 0) return lp;
  const uint32_t mask = (1u << lp) - 1u, hb = 1u << (lp - 1);
  uint32_t Pv = mask, Mv = 0;
  int score = lp;
  for (int x = 0; x < lt; ++x) {
    uint32_t Eq = eq_mask8(P, uint32_t(T >> (8 * x)) & 0xFFu) & mask;
    uint32_t Xv = Eq | Mv;
    uint32_t Xh = (((Eq & Pv) + Pv) ^ Pv) | Eq;
    uint32_t Ph = Mv | ~(Xh | Pv);
    uint32_t Mh = Pv & Xh;
    score += int((Ph & hb) != 0) - int((Mh & hb) != 0);
    Ph = (Ph << 1) | 1u;  // row 0 of the edit table grows by one per column
    Mh <<= 1;
    Pv = Mh | ~(Xv | Ph);
    Mv = Ph & Xv;
  }
  return score;
}

// Two independent lev_packed8 evaluations advanced in lockstep (each column
// step applied only while that pair's text lasts): the same results, with two
// dependency chains interleaved. Pairs with an empty string take the closed form.
__device__ __forceinline__ void lev_packed8_x2(uint64_t P0, int lp0, uint64_t T0, int lt0,
                                               uint64_t P1, int lp1, uint64_t T1, int lt1,
                                               int& d0, int& d1) {
  const uint32_t mask0 = lp0 > 0 ? (1u << lp0) - 1u : 0u, hb0 = lp0 > 0 ? 1u << (lp0 - 1) : 0u;
  const uint32_t mask1 = lp1 > 0 ? (1u << lp1) - 1u : 0u, hb1 = lp1 > 0 ? 1u << (lp1 - 1) : 0u;
  uint32_t Pv0 = mask0, Mv0 = 0, Pv1 = mask1, Mv1 = 0;
  int s0 = lp0, s1 = lp1;
  const int n = max(lp0 > 0 ? lt0 : 0, lp1 > 0 ? lt1 : 0);
  for (int x = 0; x < n; ++x) {
    const uint32_t Eq0 = eq_mask8(P0, uint32_t(T0 >> (8 * x)) & 0xFFu) & mask0;
    const uint32_t Eq1 = eq_mask8(P1, uint32_t(T1 >> (8 * x)) & 0xFFu) & mask1;
    const uint32_t Xv0 = Eq0 | Mv0, Xv1 = Eq1 | Mv1;
    const uint32_t Xh0 = (((Eq0 & Pv0) + Pv0) ^ Pv0) | Eq0;
    const uint32_t Xh1 = (((Eq1 & Pv1) + Pv1) ^ Pv1) | Eq1;
    uint32_t Ph0 = Mv0 | ~(Xh0 | Pv0), Ph1 = Mv1 | ~(Xh1 | Pv1);
    uint32_t Mh0 = Pv0 & Xh0, Mh1 = Pv1 & Xh1;
    const int e0 = int((Ph0 & hb0) != 0) - int((Mh0 & hb0) != 0);
    const int e1 = int((Ph1 & hb1) != 0) - int((Mh1 & hb1) != 0);
    Ph0 = (Ph0 << 1) | 1u;
    Ph1 = (Ph1 << 1) | 1u;
    Mh0 <<= 1;
    Mh1 <<= 1;
    if (x < lt0) {
      s0 += e0;
      Pv0 = Mh0 | ~(Xv0 | Ph0);
      Mv0 = Ph0 & Xv0;
    }
    if (x < lt1) {
      s1 += e1;
      Pv1 = Mh1 | ~(Xv1 | Ph1);
      Mv1 = Ph1 & Xv1;
    }
  }
  d0 = lp0 == 0 ? lt0 : (lt0 == 0 ? lp0 : s0);
  d1 = lp1 == 0 ? lt1 : (lt1 == 0 ? lp1 : s1);
}

// Edit distance by the textbook row recurrence, for tokens longer than 8
// bytes (bytes read from the global tables; ns, nt <= TT_MAX_TOKEN_BYTES).
__device__ int lev_rows(const uint8_t* s, int ns, const uint8_t* t, int nt) {
  if (ns > nt) {  // keep the row short
    const uint8_t* u = s; s = t; t = u;
    int n = ns; ns = nt; nt = n;
  }
  uint16_t row[TT_MAX_TOKEN_BYTES + 1];
  for (int i = 0; i <= ns; ++i) row[i] = uint16_t(i);
  for (int j = 1; j <= nt; ++j) {
    uint8_t tj = t[j - 1];
    int diag = row[0];
    row[0] = uint16_t(j);
    for (int i = 1; i <= ns; ++i) {
      int up = row[i];
      int v = min(min(up + 1, int(row[i - 1]) + 1), diag + (s[i - 1] == tj ? 0 : 1));
      diag = up;
      row[i] = uint16_t(v);
    }
  }
  return row[ns];
}

// Bytes of a K x TW tile of 4-bit cells, in whole 32-bit words (the sweep
// and the tile fill update cells through the words holding them), rounded to
// 16 bytes.
__host__ __device__ __forceinline__ size_t tile_bytes(int K, int TW) {
  return ((size_t(K) * TW + 7) / 8 * 4 + 15) & ~size_t(15);
}

struct PairSmem {
  uint64_t* tok;  // [K + M] packed bytes (valid when len <= 8)
  int32_t* diag;  // [3 * (K + 2)] rotating anti-diagonals, indexed by i
  uint32_t* path; // [K + M] backtracked cells (i << 16 | j), reverse order
  uint8_t* tile;  // [K * TW / 2] 4-bit cells, two per byte, row i at (i - 1) * tw:
                  // cost (15: 15 or more, recomputed), then direction
  uint16_t* len;  // [K + M] token byte lengths
};

__device__ __forceinline__ PairSmem carve(char* base, int K, int M, int TW) {
  PairSmem s;
  size_t off = 0;
  s.tok = reinterpret_cast<uint64_t*>(base + off);
  off += sizeof(uint64_t) * (K + M);
  s.diag = reinterpret_cast<int32_t*>(base + off);
  off += sizeof(int32_t) * 3 * (K + 2);
  s.path = reinterpret_cast<uint32_t*>(base + off);
  off += sizeof(uint32_t) * (K + M);
  s.tile = reinterpret_cast<uint8_t*>(base + off);
  off += tile_bytes(K, TW);
  s.len = reinterpret_cast<uint16_t*>(base + off);
  return s;
}

// One warp aligns pair b in its own shared-memory region.
__device__ __forceinline__ void align_pair(const AlignArgs& a, int b, char* region, int lane) {
  const int K = a.max_k, M = a.max_m, TW = a.tile_w;
  PairSmem sm = carve(region, K, M, TW);

  if (!csr_ok(a.draft_off, b, a.n_draft) || !csr_ok(a.target_off, b, a.n_target)) {
    if (lane == 0) {
      a.status[b] = TT_REQ_BAD_OFFSETS;
      if (a.path_len) a.path_len[b] = 0;
      if (a.cost) a.cost[b] = -1;
    }
    return;
  }
  const int d0 = a.draft_off[b], k = a.draft_off[b + 1] - d0;
  const int t0 = a.target_off[b], m = a.target_off[b + 1] - t0;
  if (a.excl)  // the row pass leaves these columns out of its sums
    for (int j = lane; j <= m; j += 32)
      a.excl[int64_t(t0) + b + j] = j < m ? a.target_cols[t0 + j] : -1;
  int st = 0;
  if (k == 0 || m == 0) st |= TT_REQ_EMPTY;
  if (k > K || m > M || k > TT_MAX_K || m > TT_MAX_M) st |= TT_REQ_TOO_LONG;
  if (st == 0) {
    // stage every token: length and (if <= 8 bytes) its packed bytes
    int flag = 0;
    for (int x = lane; x < k + m; x += 32) {
      const bool is_d = x < k;
      const int id = is_d ? a.draft_ids[d0 + x] : a.target_ids[t0 + x - k];
      const tt_vocab& v = is_d ? a.vd : a.vt;
      uint16_t ln = 0;
      uint64_t packed = 0;
      if (id < 0 || id >= v.n_tokens) {
        flag |= TT_REQ_ID_OUT_OF_RANGE;
      } else {
        const int64_t o0 = v.offsets[id], o1 = v.offsets[id + 1];
        const int64_t n = o1 - o0;
        if (o0 < 0 || o1 > v.n_bytes || n < 0) {
          flag |= TT_REQ_ID_OUT_OF_RANGE;
        } else if (n > TT_MAX_TOKEN_BYTES) {
          flag |= TT_REQ_TOO_LONG;
        } else {
          ln = uint16_t(n);
          if (n <= 8) {  // all loads issued before any is used
            uint8_t by[8];
#pragma unroll
            for (int y = 0; y < 8; ++y) by[y] = y < n ? v.bytes[o0 + y] : uint8_t(0);
#pragma unroll
            for (int y = 0; y < 8; ++y) packed |= uint64_t(by[y]) << (8 * y);
          }
        }
      }
      sm.len[x] = ln;
      sm.tok[x] = packed;
    }
    st = __reduce_or_sync(0xffffffffu, flag);
  }
  if (st != 0) {
    for (int j = lane; j < m; j += 32)
      if (a.map) a.map[t0 + j] = -1;
    for (int i = lane; i < k; i += 32)
      if (a.need) a.need[d0 + i] = 0;
    if (lane == 0) {
      a.status[b] = st;
      if (a.path_len) a.path_len[b] = 0;
      if (a.cost) a.cost[b] = -1;
    }
    return;
  }

  const int W0 = a.window < 0 ? k + m : max(a.window, abs(k - m));  // band half-width
  const int tw = min(m, 2 * W0 + 1);                                 // tile cells per row

  // local cost d(i, j) of draft token i and target token j (1-based)
  auto token_cost = [&](int i, int j) -> int {
    const int ld = sm.len[i - 1], lt = sm.len[k + j - 1];
    if (ld <= 8 && lt <= 8) {
      // pattern = the longer string, text = the shorter (fewer steps)
      return ld >= lt ? lev_packed8(sm.tok[i - 1], ld, sm.tok[k + j - 1], lt)
                      : lev_packed8(sm.tok[k + j - 1], lt, sm.tok[i - 1], ld);
    }
    const int di = a.draft_ids[d0 + i - 1], ti = a.target_ids[t0 + j - 1];
    return lev_rows(a.vd.bytes + a.vd.offsets[di], ld, a.vt.bytes + a.vt.offsets[ti], lt);
  };

  // 1. banded local costs, four bits each (a cost of 15 or more -- possible
  // only for tokens of more than 8 bytes -- is stored as 15 and recomputed in
  // the sweep); row i (1-based) holds j = jlo(i) .. jhi(i) at (i - 1) * tw.
  // Each lane takes the two cells of one byte per step: when both are short
  // tokens their two bit-parallel evaluations run interleaved.
  for (int q = lane; 2 * q < k * tw; q += 32) {
    int ii[2], cc[2], jj[2];
    bool ok[2];
    ii[0] = (2 * q) / tw + 1;
    cc[0] = 2 * q - (ii[0] - 1) * tw;
    ii[1] = cc[0] + 1 == tw ? ii[0] + 1 : ii[0];
    cc[1] = cc[0] + 1 == tw ? 0 : cc[0] + 1;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      jj[h] = max(1, ii[h] - W0) + cc[h];
      ok[h] = 2 * q + h < k * tw && jj[h] <= min(m, ii[h] + W0);
    }
    int d[2] = {0, 0};
    const bool short0 = ok[0] && sm.len[ii[0] - 1] <= 8 && sm.len[k + jj[0] - 1] <= 8;
    const bool short1 = ok[1] && sm.len[ii[1] - 1] <= 8 && sm.len[k + jj[1] - 1] <= 8;
    if (short0 && short1) {
      // pattern = the longer string, text = the shorter, for each pair
      uint64_t P[2], T[2];
      int lp[2], lt[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int ld = sm.len[ii[h] - 1], ltk = sm.len[k + jj[h] - 1];
        const uint64_t pd = sm.tok[ii[h] - 1], pt = sm.tok[k + jj[h] - 1];
        const bool dl = ld >= ltk;
        P[h] = dl ? pd : pt;
        lp[h] = dl ? ld : ltk;
        T[h] = dl ? pt : pd;
        lt[h] = dl ? ltk : ld;
      }
      lev_packed8_x2(P[0], lp[0], T[0], lt[0], P[1], lp[1], T[1], lt[1], d[0], d[1]);
    } else {
      if (ok[0]) d[0] = token_cost(ii[0], jj[0]);
      if (ok[1]) d[1] = token_cost(ii[1], jj[1]);
    }
    sm.tile[q] = uint8_t((ok[0] ? min(d[0], 15) : 0) | ((ok[1] ? min(d[1], 15) : 0) << 4));
  }
  __syncwarp();  // every cost is in the tile before the sweep reads it

  // A cell's cost nibble and, once its predecessor is chosen, its direction:
  // set by one XOR on the 32-bit word holding it (the other nibbles of the
  // word belong to cells of other diagonals, which other lanes may be setting).
  uint32_t* tile32 = reinterpret_cast<uint32_t*>(sm.tile);
  auto cell_of = [&](int i, int j) { return (i - 1) * tw + (j - max(1, i - W0)); };
  auto nibble = [&](int p) { return (sm.tile[p >> 1] >> ((p & 1) * 4)) & 15; };
  auto set_dir = [&](int p, int stored, int dir) {
    atomicXor(&tile32[p >> 3], uint32_t(stored ^ dir) << ((p & 7) * 4));
  };

  // 2. anti-diagonal sweep. A diagonal s = i + j holds the cells
  // i = lo(s) .. hi(s); each depends on the two diagonals before it.
  int cstar;
  if (W0 <= 31) {
    // at most W0 + 1 <= 32 cells per diagonal: lane l holds cell lo(s) + l of
    // diagonal s in a register, and the previous two diagonals' values come by
    // shuffles (a cell outside their ranges is infinite: a border, or outside
    // the band); diagonal 0 is C(0,0) = 0, diagonal 1 holds borders only
    int v1 = kInf, lo1 = 1, n1 = 0;                // diagonal s - 1
    int v2 = lane == 0 ? 0 : kInf, lo2 = 0, n2 = 1;  // diagonal s - 2
    for (int s = 2; s <= k + m; ++s) {
      const int lo = max(max(1, s - m), (s - W0 + 1) >> 1);
      const int hi = min(min(k, s - 1), (s + W0) >> 1);
      const int i = lo + lane, j = s - i;
      const int su = i - 1 - lo1, sl = i - lo1, sd = i - 1 - lo2;
      const int up0 = __shfl_sync(0xffffffffu, v1, su & 31);
      const int left0 = __shfl_sync(0xffffffffu, v1, sl & 31);
      const int dg0 = __shfl_sync(0xffffffffu, v2, sd & 31);
      int v = kInf;
      if (i <= hi) {
        const int up = (su >= 0 && su < n1) ? up0 : kInf;
        const int left = (sl >= 0 && sl < n1) ? left0 : kInf;
        int best = (sd >= 0 && sd < n2) ? dg0 : kInf, dir = 0;
        if (up < best) { best = up; dir = 1; }
        if (left < best) { best = left; dir = 2; }
        const int p = cell_of(i, j);
        const int stored = nibble(p);
        const int cost = stored == 15 ? token_cost(i, j) : stored;
        v = best >= kInf ? kInf : best + cost;
        set_dir(p, stored, dir);
      }
      v2 = v1;
      lo2 = lo1;
      n2 = n1;
      v1 = v;
      lo1 = lo;
      n1 = hi - lo + 1;
    }
    cstar = __shfl_sync(0xffffffffu, v1, (k - lo1) & 31);  // C(k, m): the last diagonal's cell k
    __syncwarp();
  } else {
    // buffer s % 3 holds C(i, s - i) at index i
    int32_t* D[3] = {sm.diag, sm.diag + (K + 2), sm.diag + 2 * (K + 2)};
    for (int i = lane; i <= k + 1; i += 32) {
      D[0][i] = i == 0 ? 0 : kInf;  // s = 0: C(0,0) = 0
      D[1][i] = kInf;               // s = 1: border cells only
    }
    __syncwarp();
    for (int s = 2; s <= k + m; ++s) {
      int32_t* cur = D[s % 3];
      const int32_t* p1 = D[(s + 2) % 3];
      const int32_t* p2 = D[(s + 1) % 3];
      const int lo = max(max(1, s - m), (s - W0 + 1) >> 1);  // ceil((s - W0) / 2)
      const int hi = min(min(k, s - 1), (s + W0) >> 1);
      for (int i = lo + lane; i <= hi; i += 32) {
        const int j = s - i;
        const int up = p1[i - 1], left = p1[i], dg = p2[i - 1];
        int best = dg, dir = 0;
        if (up < best) { best = up; dir = 1; }
        if (left < best) { best = left; dir = 2; }
        const int p = cell_of(i, j);
        const int stored = nibble(p);
        const int cost = stored == 15 ? token_cost(i, j) : stored;
        cur[i] = best >= kInf ? kInf : best + cost;
        set_dir(p, stored, dir);
      }
      if (lane == 0) {  // guards: neighbours just outside the diagonal read as infinite
        if (lo - 1 >= 0) cur[lo - 1] = kInf;
        if (hi + 1 <= k + 1) cur[hi + 1] = kInf;
      }
      __syncwarp();
    }
    cstar = D[(k + m) % 3][k];
  }

  // 3. backtrack on lane 0, from (k, m) to (1, 1)
  int L = 0;
  if (lane == 0) {
    int i = k, j = m;
    while (i > 0 && j > 0 && L < k + m) {
      sm.path[L++] = (uint32_t(i) << 16) | uint32_t(j);
      const int dir = nibble(cell_of(i, j));
      if (dir == 0) { --i; --j; }
      else if (dir == 1) { --i; }
      else { --j; }
    }
  }
  L = __shfl_sync(0xffffffffu, L, 0);
  for (int i = lane; i < k; i += 32)
    if (a.need) a.need[d0 + i] = 0;
  __syncwarp();

  // 4. outputs in forward order
  int32_t* pout = a.path ? a.path + 2 * (size_t(d0) + t0) : nullptr;
  for (int x = lane; x < L; x += 32) {
    const uint32_t cell = sm.path[L - 1 - x];
    const int i = int(cell >> 16), j = int(cell & 0xffffu);
    if (pout) {
      pout[2 * x] = i - 1;
      pout[2 * x + 1] = j - 1;
    }
    // last cell of column j on the path carries the largest i
    const bool last_in_col = x == L - 1 || int(sm.path[L - 2 - x] & 0xffffu) != j;
    if (last_in_col) {
      if (a.map) a.map[t0 + j - 1] = i - 1;
      if (a.need) a.need[d0 + i - 1] = 1;
    }
  }
  if (lane == 0) {
    a.status[b] = 0;
    if (a.path_len) a.path_len[b] = L;
    if (a.cost) a.cost[b] = cstar;
  }
}

// Before the row pass, at most one CTA per SM whose warps loop over the pairs
// (the row pass's CTAs fit beside it and stream target rows while the pairs
// are aligned); alone, one warp per pair (launch_align).
__global__ void __launch_bounds__(kAlignWarpsMax * 32, 4)
    align_kernel(AlignArgs a) {
  extern __shared__ __align__(16) char smem_raw[];
  // the row pass may start streaming target rows now; it waits for this grid
  // before it reads the needed-draft-row flags
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (a.work && blockIdx.x == 0 && threadIdx.x < kWorkShards)
    a.work[threadIdx.x * kWorkStride] = 0ull;  // read after this grid ends
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  char* region = smem_raw + size_t(warp) * a.smem_per_warp;
  for (int b = blockIdx.x * a.warps_per_block + warp; b < a.B;
       b += int(gridDim.x) * a.warps_per_block) {
    align_pair(a, b, region, lane);
    __syncwarp();  // the region is reused by the warp's next pair
  }
}

}  // namespace

size_t align_smem_per_warp(int max_k, int max_m, int tile_w) {
  size_t n = sizeof(uint64_t) * (max_k + max_m) + sizeof(int32_t) * 3 * (max_k + 2) +
             sizeof(uint32_t) * (max_k + max_m) +
             tile_bytes(max_k, tile_w) +
             sizeof(uint16_t) * (max_k + max_m);
  return (n + 15) & ~size_t(15);
}

int align_tile_width(int max_k, int max_m, int window) {
  const int W0 = window < 0 ? max_k + max_m : max(window, max(max_k, max_m) - 1);
  return min(max_m, 2 * W0 + 1);
}

cudaError_t preload_align() {
  return cudaFuncSetAttribute(align_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kAlignSmemMax);
}

cudaError_t launch_align(const AlignArgs& args, cudaStream_t stream) {
  static int n_sm[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) dev = 0;
  if (n_sm[dev] == 0 &&
      cudaDeviceGetAttribute(&n_sm[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    n_sm[dev] = 148;
  // A grid followed by the row pass (it zeroes the row pass's work counters)
  // takes at most one CTA of at most kAlignWarpsStep warps per SM, whose warps
  // loop over the pairs, so that three row-pass CTAs fit beside it and stream
  // target rows while it runs; an alignment on its own takes one warp per pair
  // and as many CTAs as fit.
  AlignArgs a = args;
  if (a.work) a.warps_per_block = std::min(a.warps_per_block, kAlignWarpsStep);
  const int per_pair = (a.B + a.warps_per_block - 1) / a.warps_per_block;
  const int blocks = a.work ? std::min(per_pair, n_sm[dev]) : per_pair;
  const size_t smem = a.smem_per_warp * size_t(a.warps_per_block);
  align_kernel<<<blocks, a.warps_per_block * 32, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace tt
