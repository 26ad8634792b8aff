// stream_order.h -- what this library last put on each CUDA stream, as far as
// the next attention call needs to know it.  Not part of the ABI.
//
// A decode grid may start without waiting for the grid before it (chain 3 in
// the attention kernel) only when that grid is one of this library's split-K
// combines: a combine releases the next grid only after its own wait, so
// every grid before it has completed by then, and the decode grid defers its
// writes of the output and the workspace (which the combine uses) until its
// own wait.  Every kernel launch and copy the library issues records itself
// here, so a sync kernel, an append or a table copy between two attention
// calls turns the start-without-waiting off for the next call.
#pragma once

// record the library's latest launch on `stream` (a combine or anything else)
void kvp_note_stream(void *stream, bool combine);
// true when the library's latest launch on `stream` was a split-K combine
bool kvp_stream_after_combine(void *stream);

// The workspace areas of a shared-prefix call whose combine was the latest
// launch on a stream.  The next shared-prefix call on the same workspace
// may then write its plan, its skips (into the other skip array) and its
// table sync while that combine still runs: the combine reads none of them.
struct KvpCascadeNote {
    const void *ws;     // workspace base
    const void *skip;   // the skip array the combine reads
    const void *flags;  // the plan kernel's flags
    const void *plan;   // the plan words
};
// mark the latest launch on `stream` (a shared-prefix call's combine) with
// its workspace areas
void kvp_note_cascade_combine(void *stream, const KvpCascadeNote &n);
// true, with *n filled in, when the latest launch on `stream` was a
// shared-prefix call's combine
bool kvp_stream_after_cascade(void *stream, KvpCascadeNote *n);
