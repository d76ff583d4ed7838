// The token list of Sec. 4.1 and Alg. 2 (token generation thread, pull
// responding threads): a queue of tokens, each the global step at which the
// batch it goes with is handed to a worker.  Token values start at 0 and each
// value repeats M times, so the i-th token handed out is floor(i / M).  (The
// paper also writes t_i = floor(i / K) with K = ceil(Q / M), which repeats each
// value K times and contradicts the sentence before it; this follows the
// sentence, which is also what a gradient buffer of capacity M needs.)
//
// Refill follows Alg. 2: under a lock, whenever the list holds fewer tokens
// than there are workers, new tokens are appended at the tail until it holds
// one per worker.  Fetching takes the head under the same lock, so any number
// of host threads may fetch concurrently.
#include <deque>
#include <mutex>
#include <new>

#include "gba.h"

struct gba_token_list {
  std::mutex mu;
  std::deque<int64_t> q;
  int64_t repeats = 1;
  int32_t workers = 1;
  int64_t next_index = 0;  // index i of the next token to generate
  int64_t fetched = 0;

  void refill() {  // caller holds mu
    while ((int64_t)q.size() < (int64_t)workers) {
      q.push_back(next_index / repeats);
      ++next_index;
    }
  }
};

extern "C" {

gba_status gba_token_list_create(int64_t repeats, int32_t workers, gba_token_list** out) {
  if (!out) return GBA_E_ARG;
  *out = nullptr;
  if (repeats < 1 || workers < 1) return GBA_E_ARG;
  gba_token_list* tl = new (std::nothrow) gba_token_list();
  if (!tl) return GBA_E_OOM;
  tl->repeats = repeats;
  tl->workers = workers;
  {
    std::lock_guard<std::mutex> lock(tl->mu);
    tl->refill();
  }
  *out = tl;
  return GBA_OK;
}

gba_status gba_fetch_token(gba_token_list* tl, int64_t* token) {
  if (!tl || !token) return GBA_E_ARG;
  std::lock_guard<std::mutex> lock(tl->mu);
  if (tl->q.empty()) tl->refill();
  *token = tl->q.front();
  tl->q.pop_front();
  ++tl->fetched;
  tl->refill();  // the fetch triggers the generation step
  return GBA_OK;
}

gba_status gba_token_list_state(gba_token_list* tl, int64_t* queued, int64_t* fetched) {
  if (!tl) return GBA_E_ARG;
  std::lock_guard<std::mutex> lock(tl->mu);
  if (queued) *queued = (int64_t)tl->q.size();
  if (fetched) *fetched = tl->fetched;
  return GBA_OK;
}

void gba_token_list_destroy(gba_token_list* tl) { delete tl; }

}  // extern "C"
