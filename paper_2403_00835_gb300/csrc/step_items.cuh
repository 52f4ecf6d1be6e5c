// Bodies of the per-iteration helpers (shared by their standalone kernels and
// the persistent per-iteration kernel); 128 threads, `sync` their barrier.
//   embed_unit  - one (row, 128-column group) of the embedding: fp32 residual
//                 stream, first RMSNorm input, the group's sum of squares
//   accept_body - Alg. 3's fixed-point test, commit and refill for sequence b
// Guesses come from a counter-based splitmix64 stream (Vigna): the
// ((b<<40 | iteration<<16 | slot) + 1)-th output for key `seed`.
#pragma once
#include "act.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace cllm {

__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t i) {
  uint64_t z = seed + i * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ int draw_guess(const AcceptArgs& a, int b, int step, int slot) {
  const uint64_t ctr = (static_cast<uint64_t>(b) << 40) | (static_cast<uint64_t>(step) << 16) |
                       static_cast<uint64_t>(slot);
  const uint64_t r = splitmix64_at(a.seed, ctr + 1) >> 32;
  if (a.guess_mode == 1) {
    const int len = a.plen[b];
    return a.prompts[static_cast<size_t>(b) * a.prompt_ld + ((r * static_cast<uint64_t>(len)) >> 32)];
  }
  return static_cast<int>((r * static_cast<uint64_t>(a.V)) >> 32);
}

template <typename Act, class Sync>
__device__ void embed_unit(const EmbedArgs& a, int t, int grp, int i, float* red, Sync sync) {
  const int m = grp * 128 + i;
  int tok, pos, b;
  if (a.block != nullptr) {
    b = t / a.n;
    const int k = t - b * a.n;
    tok = a.block[b * a.n + k];
    pos = a.L[b] + k;
  } else {
    tok = a.tok_in[t];
    pos = a.pos_in[t];
    b = a.bidx_in[t];
  }
  if (tok < 0 || tok >= a.V) {
    if (i == 0 && grp == 0) atomicOr(a.err, DERR_TOKEN);
    tok = 0;
  }
  const float e = ld_act(static_cast<const Act*>(a.emb), static_cast<size_t>(tok) * a.d + m);
  const size_t o = static_cast<size_t>(t) * a.d + m;
  a.x[o] = e;
  st_gin(static_cast<Act*>(a.xg), o, a.plane, e * ld_act(static_cast<const Act*>(a.gain), m));
  const float s = warp_sum(e * e);
  if ((i & 31) == 0) red[i >> 5] = s;
  sync();
  if (i == 0) a.ssq[static_cast<size_t>(grp) * a.ldt + t] = ((red[0] + red[1]) + red[2]) + red[3];
  if (grp == 0 && i == 0) {
    if (pos < 0 || pos >= a.max_seq) atomicOr(a.err, DERR_CAPACITY);
    a.pos[t] = pos;
    a.bidx[t] = b;
  }
  if (a.block != nullptr && t == 0 && grp == 0) {
    for (int bb = i; bb < a.B; bb += 128) {
      a.seq_start[bb] = a.L[bb];
      a.seq_row0[bb] = bb * a.n;
      a.seq_nrows[bb] = a.n;
    }
  }
  sync();  // red[] is reused by the next unit
}

// Acceptance statistics of one iteration of sequence b (decode loop): the
// block y of active width w commits acc tokens at positions c..c+acc-1,
// c = tokens committed so far.  Fast-forwarded count (Table 3): acc itself,
// the head included.  Stationary tokens (Sec. 3.3): a position is
// stationary when, before it is committed, it already holds its final token
// while an earlier slot of the block is wrong, and keeps that token in every
// later block until it is committed.  Kept online: a slot's candidate flag
// is set when it holds an unchanged value at an iteration whose accepted
// prefix ends before it, and restarts whenever its value changes; a committed
// token is final, so a committed position is stationary exactly when its flag
// is set.  Windows: a window opens with the first block that starts at or
// after the previous window's end and covers that block's w positions;
// stationary positions count toward the window that holds them.
__device__ inline void accept_stats(const AcceptArgs& a, int b, const int* y, int w, int acc) {
  const int n = a.n;
  const int c = a.committed[b];
  int* pos = a.st_pos + static_cast<size_t>(b) * n;
  int* val = a.st_val + static_cast<size_t>(b) * n;
  int* cand = a.st_cand + static_cast<size_t>(b) * n;
  if (c >= a.win_end[b]) {
    if (a.win_end[b] > 0) atomicAdd(&a.win_hist[min(a.win_cnt[b], n)], 1ull);
    a.win_end[b] = c + w;
    a.win_cnt[b] = 0;
    atomicAdd(&a.totals[0], 1ull);
  }
  atomicAdd(&a.acc_hist[min(acc, n)], 1ull);
  for (int k = 0; k < w; ++k) {
    const int p = c + k, q = p % n;
    const int later = k > acc ? 1 : 0;
    if (pos[q] != p || val[q] != y[k]) {
      pos[q] = p;
      val[q] = y[k];
      cand[q] = later;
    } else {
      cand[q] |= later;
    }
  }
  int found = 0;
  for (int k = 0; k < acc; ++k) {
    const int p = c + k, q = p % n;
    if (cand[q] && p < a.win_end[b]) ++found;
    pos[q] = -1;  // committed: the slot's next position starts afresh
  }
  if (found) {
    a.win_cnt[b] += found;
    atomicAdd(&a.totals[1], static_cast<unsigned long long>(found));
  }
}

template <class Sync>
__device__ void accept_body(const AcceptArgs& a, int b, int* s_act, int* s_com, Sync sync) {
  int active = 0, committed_now = 0;
  if (b < a.B) {
    const int n = a.n;
    const int* P = a.pred + b * n;
    int* y = a.block + b * n;
    if (!(a.decode && a.done[b])) {
      const int w = (a.decode && a.shrink) ? a.width[b] : n;  // active rows of the block
      if (a.decode && a.traj != nullptr && a.iters[b] < a.traj_cap) {
        int* tr = a.traj + (static_cast<size_t>(a.iters[b]) * a.B + b) * n;
        for (int k = 0; k < n; ++k) tr[k] = k < w ? y[k] : -1;
      }
      int acc = 1;
      while (acc < w && y[acc] == P[acc - 1]) ++acc;
      if (a.decode) {
        bool stop = false;
        if (a.eos >= 0) {
          for (int k = 0; k < acc; ++k)
            if (y[k] == a.eos) {
              acc = k + 1;
              stop = true;
              break;
            }
        }
        const int room = a.max_new - a.committed[b];
        if (acc > room) acc = room;
        if (a.acc_hist != nullptr) accept_stats(a, b, y, w, acc);
        int* out = a.out + static_cast<size_t>(b) * a.max_new + a.committed[b];
        for (int k = 0; k < acc; ++k) out[k] = y[k];
        a.committed[b] += acc;
        a.iters[b] += 1;
        if (stop || a.committed[b] >= a.max_new) a.done[b] = 1;
        active = a.done[b] ? 0 : 1;
        committed_now = acc;
      }
      a.accepted[b] = acc;
      a.L[b] += acc;
      a.head[b] = P[acc - 1];
      if (a.decode && !a.shrink) {
        // next block: the predictions from the new head on, then fresh guesses
        const int keep = n - acc + 1;
        const int step = a.iters[b];
        for (int k = 0; k < n; ++k) y[k] = (k < keep) ? P[acc - 1 + k] : draw_guess(a, b, step, k);
        if (a.pool != nullptr) {
          // lookahead (Sec. 3.3): the pooled continuation of the new head,
          // from earlier iterations, fills slots 1..; then this iteration's
          // n-grams (key P[k], value P[k+1..k+pool_w], k ascending) enter
          // (a prediction outside the vocabulary -- only after a device
          // error -- is never used as a key)
          int* pb = a.pool + static_cast<size_t>(b) * a.V * a.pool_w;
          const int h = P[acc - 1];
          if (static_cast<unsigned>(h) < static_cast<unsigned>(a.V)) {
            const int* cand = pb + static_cast<size_t>(h) * a.pool_w;
            if (cand[0] >= 0) {
              const int w = min(a.pool_w, n - 1);
              for (int j = 0; j < w; ++j) y[1 + j] = cand[j];
            }
          }
          for (int k = 0; k + a.pool_w < n; ++k) {
            if (static_cast<unsigned>(P[k]) >= static_cast<unsigned>(a.V)) continue;
            int* dst = pb + static_cast<size_t>(P[k]) * a.pool_w;
            for (int j = 0; j < a.pool_w; ++j) dst[j] = P[k + 1 + j];
          }
        }
      } else if (a.decode) {
        const int step = a.iters[b];
        if (acc == w) {
          // the whole window is fixed: a fresh block, the new head then guesses
          for (int k = 0; k < n; ++k) y[k] = (k == 0) ? P[acc - 1] : draw_guess(a, b, step, k);
          a.width[b] = n;
        } else {
          // the window narrows to the positions not yet fixed; rows beyond it
          // are computed but ignored (they hold valid tokens)
          for (int k = 0; k < n; ++k) y[k] = P[min(acc - 1 + k, n - 1)];
          a.width[b] = w - acc;
        }
      }
    }
  }
  int wa = active, wc = committed_now;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    wa += __shfl_xor_sync(0xffffffffu, wa, o);
    wc += __shfl_xor_sync(0xffffffffu, wc, o);
  }
  if ((b & 31) == 0) {
    s_act[b >> 5] = wa;
    s_com[b >> 5] = wc;
  }
  sync();
  if (b == 0) {
    a.status[0] = s_act[0] + s_act[1] + s_act[2] + s_act[3];
    a.status[1] = s_com[0] + s_com[1] + s_com[2] + s_com[3];
  }
}


}  // namespace cllm
